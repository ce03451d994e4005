// index_kernels.cu -- integer bookkeeping of the homogenized step and row gathers.
//
// The prepass turns the op stream into every index the state kernels use, so the time
// loop itself never branches on an op (Algorithm 1 has no op-dependent branch):
//   p_traj[t]   pointer before step t: p_0 = 0, p_{t+1} = p_t + op_t (Sec. 3);
//   top[t]      history index of the state at slot p_t at time t: 0 is the initial state,
//               tau + 1 the state step tau wrote. Step t reads history row top[t];
//   slot_last   history index last written to each slot after the last step (-1: never).
// Every step writes slot p_t + 1 (Algorithm 1), which in history terms is row t + 1.
#include <algorithm>
#include <map>
#include <mutex>

#include "common.cuh"

namespace sl {
namespace {

constexpr int kPrepassThreads = 32;
// shared-memory staging of prepass_walk_vec_kernel: four [32][32] int32 blocks and the ops
constexpr size_t kWalkStageBytes = 4 * 32 * 32 * 4 + 32 * 32;

// One thread per instance, walking its steps in order with the instance's stack of slot
// tags. This kernel keeps the stack in a global [T+1][B] scratch (coalesced: slot-major)
// for sequences too long for shared memory and for the allocation-free entry point;
// prepass_walk_kernel below keeps it in a column of shared memory (slot-major, so the 32
// threads of a warp hit 32 distinct banks).
__global__ void __launch_bounds__(kPrepassThreads)
prepass_kernel(int T, int B, const int8_t *__restrict__ ops, int32_t *__restrict__ p_traj,
               int32_t *__restrict__ top, int32_t *__restrict__ slot_last,
               int32_t *__restrict__ gscratch, int32_t *__restrict__ err)
{
    const int lane = threadIdx.x;
    const int b = blockIdx.x * kPrepassThreads + lane;
    if (b >= B) return;
    auto tag = [&](int slot) -> int32_t & { return gscratch[(size_t)slot * B + b]; };
    tag(0) = 0;
    for (int slot = 1; slot <= T; ++slot) tag(slot) = -1;
    int p = 0, e = SL_OK;
    // the ops of 8 steps are loaded before they are used, so that the loads do not wait on
    // one another
    int8_t opq[8];
    for (int t = 0; t < T; ++t) {
        if ((t & 7) == 0)
#pragma unroll
            for (int i = 0; i < 8; ++i) opq[i] = t + i < T ? ops[(size_t)(t + i) * B + b] : 0;
        int op = opq[t & 7];
        if (op < -1 || op > 1) {  // recorded, then run as a hold so indices stay in range
            if (e == SL_OK) e = SL_ERR_OP;
            op = 0;
        }
        if (p + op < 0) {
            if (e == SL_OK) e = SL_ERR_UNDERFLOW;
            op = 0;
        }
        p_traj[(size_t)t * B + b] = p;
        top[(size_t)t * B + b] = tag(p);
        tag(p + 1) = t + 1;  // Algorithm 1: every step writes slot p + 1
        p += op;
    }
    p_traj[(size_t)T * B + b] = p;
    top[(size_t)T * B + b] = tag(p);
    for (int slot = 0; slot <= T; ++slot) slot_last[(size_t)slot * B + b] = tag(slot);
    if (e != SL_OK) atomicCAS(err, 0, e);
}

// The push-only mode's virtual timeline (compact_kernel below), when the walk builds it.
struct VirtOut {
    int32_t *vtop, *vy, *vslot, *xidx, *vstep, *kmax;
};
// (both walks also write the caller's final pointers, p_final, when it is given)

// The same walk as prepass_kernel with the slot-tag stack in shared memory, its ops loaded
// 32 steps ahead. With kPush it also builds the push-only mode's virtual timeline in the
// same walk (what compact_kernel computes from the prepass's outputs), its real-to-virtual
// index map in shared memory beside the slot tags. (Batches of whole 32-instance blocks
// take prepass_walk_vec_kernel below.)
template <bool kPush>
__global__ void __launch_bounds__(kPrepassThreads)
prepass_walk_kernel(int T, int B, const int8_t *__restrict__ ops, int32_t *__restrict__ p_traj,
                    int32_t *__restrict__ top, int32_t *__restrict__ slot_last, int32_t *__restrict__ err, VirtOut v,
                    int32_t *__restrict__ p_final)
{
    constexpr int kBlk = 32;
    extern __shared__ int32_t s_tag[];  // [T + 1][32] slot tags, then (kPush) [T + 1][32] vmap
    const int lane = threadIdx.x;
    const int b = blockIdx.x * kPrepassThreads + lane;
    if (b >= B) return;
    int32_t *s_vmap = s_tag + (size_t)(T + 1) * kPrepassThreads;
    auto tag = [&](int slot) -> int32_t & { return s_tag[slot * kPrepassThreads + lane]; };
    // virtual index of the state at real history index j (-1: a write no step reads)
    auto vmap = [&](int j) -> int32_t & { return s_vmap[j * kPrepassThreads + lane]; };
    tag(0) = 0;
    for (int slot = 1; slot <= T; ++slot) tag(slot) = -1;
    if (kPush) {
        vmap(0) = 0;
        for (int sl = 0; sl <= T; ++sl) v.vslot[(size_t)sl * B + b] = sl == 0 ? 0 : -1;
    }
    auto load = [&](int t0, int (&q)[kBlk]) {
#pragma unroll
        for (int i = 0; i < kBlk; ++i) q[i] = t0 + i < T ? (int)ops[(size_t)(t0 + i) * B + b] : 0;
    };
    int cur[kBlk], nxt[kBlk];
    load(0, cur);
    int p = 0, e = SL_OK, k = 0;
    for (int t0 = 0; t0 < T; t0 += kBlk) {
        if (t0 + kBlk < T) load(t0 + kBlk, nxt);
#pragma unroll
        for (int i = 0; i < kBlk; ++i) {
            const int t = t0 + i;
            if (t >= T) break;
            int op = cur[i];
            if (op < -1 || op > 1) {  // recorded, then run as a hold so indices stay in range
                if (e == SL_OK) e = SL_ERR_OP;
                op = 0;
            }
            if (p + op < 0) {
                if (e == SL_OK) e = SL_ERR_UNDERFLOW;
                op = 0;
            }
            const size_t ti = (size_t)t * B + b;
            const int tp = tag(p);
            p_traj[ti] = p;
            top[ti] = tp;
            tag(p + 1) = t + 1;  // Algorithm 1: every step writes slot p + 1
            if (kPush) {
                // a state that is read is a push write or the initial state (clamp never applies)
                const int rd = max(0, vmap(tp));
                v.vy[ti] = rd;
                if (op == 1) {
                    v.xidx[(size_t)k * B + b] = t;
                    v.vtop[(size_t)k * B + b] = rd;
                    v.vstep[ti] = k;
                    vmap(t + 1) = k + 1;
                    v.vslot[(size_t)(p + 1) * B + b] = k + 1;
                    ++k;
                } else {
                    v.vstep[ti] = -1;
                    vmap(t + 1) = -1;
                }
            }
            p += op;
        }
#pragma unroll
        for (int i = 0; i < kBlk; ++i) cur[i] = nxt[i];
    }
    const int tp = tag(p);
    p_traj[(size_t)T * B + b] = p;
    top[(size_t)T * B + b] = tp;
    if (p_final) p_final[b] = p;
    for (int slot = 0; slot <= T; ++slot) slot_last[(size_t)slot * B + b] = tag(slot);
    if (kPush) {
        v.vy[(size_t)T * B + b] = max(0, vmap(tp));
        for (int kk = k; kk < T; ++kk) {
            v.xidx[(size_t)kk * B + b] = -1;
            v.vtop[(size_t)kk * B + b] = 0;
        }
        v.vtop[(size_t)T * B + b] = 0;
        atomicMax(v.kmax, k);
    }
    if (e != SL_OK) atomicCAS(err, 0, e);
}

// prepass_walk_kernel for batches of whole 32-instance blocks (B % 32 == 0, ops 4-byte
// aligned), its global traffic in 16-byte pieces: the walk costs about as much per memory
// instruction of the block's one warp as per step, so the warp loads a block of 32 steps'
// ops as 4-byte words (eight lanes a row) into shared memory, walks it there, stages the
// block's pointers and tops (and virtual indices) in shared memory, and writes them four
// rows per instruction; the slot tags go out the same way, and the push-only tables that
// are mostly -1 / 0 are written so before the walk (__syncwarp orders those stores before
// the walk's own stores to the same rows).
template <bool kPush>
__global__ void __launch_bounds__(kPrepassThreads)
prepass_walk_vec_kernel(int T, int B, const int8_t *__restrict__ ops, int32_t *__restrict__ p_traj,
                        int32_t *__restrict__ top, int32_t *__restrict__ slot_last, int32_t *__restrict__ err,
                        VirtOut v, int32_t *__restrict__ p_final)
{
    constexpr int kBlk = 32;
    // [T + 1][32] slot tags, (kPush) [T + 1][32] vmap, then the block staging:
    // pointer, top, (kPush) vy, vstep, each [32 steps][32], and the ops [32 steps][32 bytes]
    extern __shared__ int32_t s_tag[];
    const int lane = threadIdx.x, b0 = blockIdx.x * kPrepassThreads, b = b0 + lane;
    const int rq = lane >> 3, pc = 4 * (lane & 7);  // row of four, 16-byte piece: the vector pattern
    int32_t *s_vmap = s_tag + (size_t)(T + 1) * kPrepassThreads;
    int32_t *st_p = s_tag + (size_t)(kPush ? 2 : 1) * (T + 1) * kPrepassThreads;
    int32_t *st_t = st_p + kBlk * 32, *st_y = st_t + kBlk * 32, *st_v = st_y + kBlk * 32;
    uint32_t *st_o = (uint32_t *)(st_v + kBlk * 32);  // [32 steps][8 words]
    auto tag = [&](int slot) -> int32_t & { return s_tag[slot * kPrepassThreads + lane]; };
    auto vmap = [&](int j) -> int32_t & { return s_vmap[j * kPrepassThreads + lane]; };
    // rows [r0, r1) of a [rows][B] int32 table: this block's 32 columns, four rows at a time
    auto fill = [&](int32_t *dst, int r0, int r1, int val) {
        const uint4 w = make_uint4(val, val, val, val);
        for (int r = r0 + rq; r < r1; r += 4) *(uint4 *)(dst + (size_t)r * B + b0 + pc) = w;
    };
    auto flush = [&](int32_t *dst, const int32_t *src, int r0, int nrows) {  // src: [nrows][32]
        for (int r = rq; r < nrows; r += 4) *(uint4 *)(dst + (size_t)(r0 + r) * B + b0 + pc) = *(const uint4 *)(src + r * 32 + pc);
    };
    auto load = [&](int t0, uint32_t (&q)[8]) {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int t = t0 + rq + 4 * j;
            q[j] = t < T ? *(const uint32_t *)(ops + (size_t)t * B + b0 + pc) : 0u;
        }
    };
    tag(0) = 0;
    for (int slot = 1; slot <= T; ++slot) tag(slot) = -1;
    if (kPush) {
        vmap(0) = 0;
        fill(v.vslot, 0, 1, 0);
        fill(v.vslot, 1, T + 1, -1);
        fill(v.xidx, 0, T, -1);
        fill(v.vtop, 0, T + 1, 0);
        __syncwarp();
    }
    uint32_t cur[8], nxt[8];
    load(0, cur);
    int p = 0, e = SL_OK, k = 0;
    for (int t0 = 0; t0 < T; t0 += kBlk) {
        if (t0 + kBlk < T) load(t0 + kBlk, nxt);
#pragma unroll
        for (int j = 0; j < 8; ++j) st_o[(rq + 4 * j) * 8 + (lane & 7)] = cur[j];
        __syncwarp();
        const int n = min(kBlk, T - t0);
        const int8_t *ob = (const int8_t *)st_o;
        for (int i = 0; i < n; ++i) {
            const int t = t0 + i;
            int op = ob[i * 32 + lane];
            if (op < -1 || op > 1) {  // recorded, then run as a hold so indices stay in range
                if (e == SL_OK) e = SL_ERR_OP;
                op = 0;
            }
            if (p + op < 0) {
                if (e == SL_OK) e = SL_ERR_UNDERFLOW;
                op = 0;
            }
            const int tp = tag(p);
            st_p[i * 32 + lane] = p;
            st_t[i * 32 + lane] = tp;
            tag(p + 1) = t + 1;  // Algorithm 1: every step writes slot p + 1
            if (kPush) {
                // a state that is read is a push write or the initial state (clamp never applies)
                const int rd = max(0, vmap(tp));
                st_y[i * 32 + lane] = rd;
                st_v[i * 32 + lane] = op == 1 ? k : -1;
                vmap(t + 1) = op == 1 ? k + 1 : -1;
                if (op == 1) {
                    v.xidx[(size_t)k * B + b] = t;
                    v.vtop[(size_t)k * B + b] = rd;
                    v.vslot[(size_t)(p + 1) * B + b] = k + 1;
                    ++k;
                }
            }
            p += op;
        }
        __syncwarp();
        flush(p_traj, st_p, t0, n);
        flush(top, st_t, t0, n);
        if (kPush) {
            flush(v.vy, st_y, t0, n);
            flush(v.vstep, st_v, t0, n);
        }
        __syncwarp();  // the staging is read before the next block overwrites it
#pragma unroll
        for (int j = 0; j < 8; ++j) cur[j] = nxt[j];
    }
    const int tp = tag(p);
    p_traj[(size_t)T * B + b] = p;
    top[(size_t)T * B + b] = tp;
    if (p_final) p_final[b] = p;
    if (kPush) {
        v.vy[(size_t)T * B + b] = max(0, vmap(tp));
        atomicMax(v.kmax, k);
    }
    __syncwarp();
    flush(slot_last, s_tag, 0, T + 1);
    if (e != SL_OK) atomicCAS(err, 0, e);
}

// out[r] = hist row (idx[r], r % B), or zeros where idx[r] < 0. E is the raw element
// bit pattern (uint32_t for float, uint16_t for bf16): a pure copy.
template <typename E>
__global__ void gather_rows_kernel(const int32_t *__restrict__ idx, int B, size_t rows, int row_elems,
                                   const E *__restrict__ hist, E *__restrict__ out)
{
    const size_t total = rows * (size_t)row_elems;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < total;
         e += (size_t)gridDim.x * blockDim.x) {
        const size_t r = e / row_elems;
        const int k = (int)(e - r * row_elems);
        const int src = idx[r];
        const int b = (int)(r % B);
        out[e] = src >= 0 ? hist[((size_t)src * B + b) * row_elems + k] : (E)0;
    }
}

// Seed the gradient history with the loss terms before the reverse loop:
// d_top_h goes to the final top, dy_t to the top after step t (Algorithm 1's output).
// One thread per (b, j); its additions run in a fixed order (final top, then t = T-1..0).
__global__ void seed_grads_kernel(int T, int B, int H, const int32_t *__restrict__ top,
                                  const float *__restrict__ d_top_h, const float *__restrict__ dy,
                                  float *__restrict__ dhist_h)
{
    const size_t n = (size_t)B * H;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n;
         e += (size_t)gridDim.x * blockDim.x) {
        const int b = (int)(e / H), j = (int)(e - (size_t)b * H);
        if (d_top_h) {
            const int s = top[(size_t)T * B + b];
            dhist_h[((size_t)s * B + b) * H + j] += d_top_h[e];
        }
        if (dy)
            for (int t = T - 1; t >= 0; --t) {
                const int s = top[(size_t)(t + 1) * B + b];
                dhist_h[((size_t)s * B + b) * H + j] += dy[(size_t)t * n + e];
            }
    }
}

// The same seeding with per-step gradients dy, for one instance and 32 units per block:
// the T + 1 rows' sums of those units accumulate in shared memory in the same order as
// above (final top, then t = T-1..0), then every row is written once. The gradient
// history is zero before the seeding, so writing the sums equals adding them.
__global__ void __launch_bounds__(32) seed_grads_dy_kernel(int T, int B, int H, const int32_t *__restrict__ top,
                                                            const float *__restrict__ d_top_h,
                                                            const float *__restrict__ dy, float *__restrict__ dhist_h)
{
    extern __shared__ float acc[];  // [T + 1][32]
    const int b = blockIdx.x, lane = threadIdx.x, j = blockIdx.y * 32 + lane;
    for (int s = 0; s <= T; ++s) acc[s * 32 + lane] = 0.0f;
    __syncwarp();
    if (j < H) {
        const size_t n = (size_t)B * H, e = (size_t)b * H + j;
        if (d_top_h) acc[top[(size_t)T * B + b] * 32 + lane] += d_top_h[e];
#pragma unroll 8
        for (int t = T - 1; t >= 0; --t) acc[top[(size_t)(t + 1) * B + b] * 32 + lane] += dy[(size_t)t * n + e];
        for (int s = 0; s <= T; ++s) dhist_h[((size_t)s * B + b) * H + j] = acc[s * 32 + lane];
    }
}

// Push-only mode: the virtual timeline of each instance. By Observation 2 of Sec. 3 only
// a push step's write is ever read (a pop or hold writes slot p + 1 above the new top,
// and the next push overwrites it before the pointer gets there), so instance b's
// computation is the chain of its push steps alone: virtual step k is its k-th push, it
// reads the virtual state of the push that wrote the slot it reads (or the initial state,
// virtual index 0) and writes virtual history row k + 1. One thread per instance walks its
// steps in order, so every index it looks up was set at an earlier step. Virtual steps
// past an instance's last push read the initial state and their writes are never read.
// A step is a push when its pointer moves up by one (ops the prepass rejected ran as
// holds). vslot is the stack of Sec. 2's definition: each slot's last pushed state.
// kmax (zero on entry) receives the most pushes of any instance.
template <bool kOnChip>
__global__ void __launch_bounds__(kPrepassThreads)
compact_kernel(int T, int B, const int32_t *__restrict__ p_traj, const int32_t *__restrict__ top,
               int32_t *__restrict__ vtop, int32_t *__restrict__ gvmap,
               int32_t *__restrict__ vy, int32_t *__restrict__ vslot, int32_t *__restrict__ xidx,
               int32_t *__restrict__ vstep, int32_t *__restrict__ kmax)
{
    extern __shared__ int32_t s_vmap[];
    const int lane = threadIdx.x, b = blockIdx.x * kPrepassThreads + lane;
    if (b >= B) return;
    // vmap: the virtual index of the state at real history index j (written at step j - 1,
    // or the initial state at j = 0), -1 for a non-push write; in shared memory when it fits
    auto vmap = [&](int j) -> int32_t & {
        return kOnChip ? s_vmap[j * kPrepassThreads + lane] : gvmap[(size_t)j * B + b];
    };
    // a state that is read is always a push write or the initial state, so the clamp never
    // applies to valid prepass output
    auto vof = [&](int j) { return max(0, vmap(j)); };
    vmap(0) = 0;
    vslot[b] = 0;  // slot 0: the initial state
    for (int sl = 1; sl <= T; ++sl) vslot[(size_t)sl * B + b] = -1;
    int k = 0;
    // the tops and pointers of 8 steps are loaded before they are used
    int tq[8], pq[9];
    for (int t = 0; t < T; ++t) {
        if ((t & 7) == 0) {
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                tq[i] = t + i < T ? top[(size_t)(t + i) * B + b] : 0;
                pq[i] = t + i <= T ? p_traj[(size_t)(t + i) * B + b] : 0;
            }
            pq[8] = t + 8 <= T ? p_traj[(size_t)(t + 8) * B + b] : 0;
        }
        const size_t i = (size_t)t * B + b;
        const int rd = vof(tq[t & 7]);
        vy[i] = rd;
        if (pq[(t & 7) + 1] - pq[t & 7] == 1) {
            xidx[(size_t)k * B + b] = t;
            vtop[(size_t)k * B + b] = rd;
            vstep[i] = k;
            vmap(t + 1) = k + 1;
            vslot[(size_t)(pq[t & 7] + 1) * B + b] = k + 1;
            ++k;
        } else {
            vstep[i] = -1;
            vmap(t + 1) = -1;
        }
    }
    vy[(size_t)T * B + b] = vof(top[(size_t)T * B + b]);
    for (int kk = k; kk < T; ++kk) {
        xidx[(size_t)kk * B + b] = -1;
        vtop[(size_t)kk * B + b] = 0;
    }
    vtop[(size_t)T * B + b] = 0;
    atomicMax(kmax, k);
}

// Push-only mode: dx rows of the steps that do not push are zero (a state no step reads
// has zero gradient); the push rows are written by the input-gradient contraction.
// A warp per row: the row's step index is read once, its 16-byte pieces written by the
// warp's lanes side by side.
__global__ void zero_nonpush_rows_kernel(size_t rows, int I4, const int32_t *__restrict__ vstep,
                                         float4 *__restrict__ dx)
{
    const int lane = threadIdx.x & 31;
    const size_t warps = (size_t)gridDim.x * (blockDim.x >> 5);
    for (size_t r = (size_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); r < rows; r += warps) {
        if (vstep[r] >= 0) continue;
        float4 *row = dx + r * I4;
        for (int i = lane; i < I4; i += 32) row[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
}

}  // namespace

cudaError_t launch_compact(stacklstm *s)
{
    if (s->walk_built_virtual) return cudaSuccess;  // the prepass's walk built the timeline
    cudaError_t e = cudaMemsetAsync(s->kmax, 0, sizeof(int32_t), s->stream);
    if (e) return e;
    // the index table on chip when the prepass's slot-tag stack is (the same size)
    const unsigned grid = ceil_div(s->B, kPrepassThreads);
    if (s->prepass_smem > 0) {
        if (s->prepass_smem > 48 * 1024 &&
            (e = smem_at_least((const void *)compact_kernel<true>, (size_t)s->prepass_smem)))
            return e;
        compact_kernel<true><<<grid, kPrepassThreads, s->prepass_smem, s->stream>>>(
            s->T, s->B, s->p_traj, s->top, s->vtop, s->vmap, s->vy, s->vslot, s->xidx, s->vstep, s->kmax);
    } else {
        compact_kernel<false><<<grid, kPrepassThreads, 0, s->stream>>>(
            s->T, s->B, s->p_traj, s->top, s->vtop, s->vmap, s->vy, s->vslot, s->xidx, s->vstep, s->kmax);
    }
    s->launches += 1;
    return cudaGetLastError();
}

cudaError_t read_virtual_steps(stacklstm *s)
{
    cudaError_t e = cudaMemcpyAsync(s->kmax_host, s->kmax, sizeof(int32_t), cudaMemcpyDeviceToHost, s->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s->stream);
    if (e) return e;
    // at least one step, so that every kernel has work of its usual shape (a batch with no
    // push at all runs one virtual step whose write nobody reads)
    s->Tr = std::max(1, std::min(s->T, (int)*s->kmax_host));
    return cudaSuccess;
}

cudaError_t launch_zero_nonpush_rows(stacklstm *s, float *dx)
{
    if (!dx) return cudaSuccess;
    const size_t rows = (size_t)s->T * s->B;
    const int I4 = s->I / 4;  // the bf16 path has I % 8 == 0
    const unsigned grid = (unsigned)std::max<size_t>(1, std::min<size_t>(ceil_div(rows, 8), (size_t)s->num_sms * 16));
    zero_nonpush_rows_kernel<<<grid, 256, 0, s->stream>>>(rows, I4, s->vstep, (float4 *)dx);
    s->launches += 1;
    return cudaGetLastError();
}

cudaError_t smem_at_least(const void *fn, size_t bytes)
{
    static std::mutex m;
    static std::map<std::pair<int, const void *>, size_t> set;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e) return e;
    std::lock_guard<std::mutex> lk(m);
    size_t &cur = set[{dev, fn}];
    if (bytes <= cur) return cudaSuccess;
    if ((e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes))) return e;
    cur = bytes;
    return cudaSuccess;
}

// The slot-tag stack goes on chip when (T + 1) slots x 32 instances fit in shared memory.
cudaError_t configure_prepass(stacklstm *s)
{
    const size_t bytes = (size_t)(s->T + 1) * kPrepassThreads * sizeof(int32_t);
    int optin = 0;
    cudaError_t e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, s->device);
    if (e) return e;
    s->prepass_smem = 0;
    s->walk_push_smem = 0;
    if (bytes + kWalkStageBytes + 1024 <= (size_t)optin) {
        if ((e = smem_at_least((const void *)prepass_walk_kernel<false>, bytes)) ||
            (e = smem_at_least((const void *)prepass_walk_vec_kernel<false>, bytes + kWalkStageBytes)))
            return e;
        s->prepass_smem = (int)bytes;
        // the push-only walk keeps the real-to-virtual index map beside the slot tags
        if (2 * bytes + kWalkStageBytes + 1024 <= (size_t)optin) {
            if ((e = smem_at_least((const void *)prepass_walk_kernel<true>, 2 * bytes)) ||
                (e = smem_at_least((const void *)prepass_walk_vec_kernel<true>, 2 * bytes + kWalkStageBytes)))
                return e;
            s->walk_push_smem = (int)(2 * bytes);
        }
    }
    return cudaSuccess;
}

cudaError_t launch_prepass(stacklstm *s, const int8_t *ops, int32_t *p_final)
{
    const unsigned grid = ceil_div(s->B, kPrepassThreads);
    s->walk_built_virtual = 0;
    s->pfinal_written = s->prepass_smem > 0;  // the walks write it; prepass_kernel does not
    // whole 32-instance blocks and word-aligned ops: the walk's traffic in 16-byte pieces
    const bool vec = s->B % kPrepassThreads == 0 && ((uintptr_t)ops & 3) == 0;
    if (s->push_only && s->walk_push_smem > 0) {
        cudaError_t e = cudaMemsetAsync(s->kmax, 0, sizeof(int32_t), s->stream);
        if (e) return e;
        const VirtOut v{s->vtop, s->vy, s->vslot, s->xidx, s->vstep, s->kmax};
        if (vec)
            prepass_walk_vec_kernel<true><<<grid, kPrepassThreads, s->walk_push_smem + kWalkStageBytes, s->stream>>>(
                s->T, s->B, ops, s->p_traj, s->top, s->slot_last, s->err, v, p_final);
        else
            prepass_walk_kernel<true><<<grid, kPrepassThreads, s->walk_push_smem, s->stream>>>(
                s->T, s->B, ops, s->p_traj, s->top, s->slot_last, s->err, v, p_final);
        s->walk_built_virtual = 1;
    } else if (s->prepass_smem > 0) {
        if (vec)
            prepass_walk_vec_kernel<false><<<grid, kPrepassThreads, s->prepass_smem + kWalkStageBytes, s->stream>>>(
                s->T, s->B, ops, s->p_traj, s->top, s->slot_last, s->err, VirtOut{}, p_final);
        else
            prepass_walk_kernel<false><<<grid, kPrepassThreads, s->prepass_smem, s->stream>>>(
                s->T, s->B, ops, s->p_traj, s->top, s->slot_last, s->err, VirtOut{}, p_final);
    } else {
        prepass_kernel<<<grid, kPrepassThreads, 0, s->stream>>>(s->T, s->B, ops, s->p_traj, s->top, s->slot_last,
                                                                s->slot_scratch, s->err);
    }
    s->launches += 1;
    return cudaGetLastError();
}

cudaError_t launch_gather_rows(stacklstm *s, const int32_t *idx, int rows, size_t elem_bytes,
                               const void *hist, void *out, int row_elems)
{
    const size_t total = (size_t)rows * row_elems;
    const unsigned grid = (unsigned)std::min<size_t>(ceil_div(total, 256), (size_t)s->num_sms * 16);
    if (total == 0) return cudaSuccess;
    if (elem_bytes == 4)
        gather_rows_kernel<uint32_t><<<grid, 256, 0, s->stream>>>(
            idx, s->B, rows, row_elems, (const uint32_t *)hist, (uint32_t *)out);
    else
        gather_rows_kernel<uint16_t><<<grid, 256, 0, s->stream>>>(
            idx, s->B, rows, row_elems, (const uint16_t *)hist, (uint16_t *)out);
    s->launches += 1;
    return cudaGetLastError();
}

cudaError_t launch_seed_grads(stacklstm *s, const float *d_top_h, const float *dy)
{
    if (!d_top_h && !dy) return cudaSuccess;
    const int32_t *top = s->push_only ? s->vy : s->top;
    const size_t acc_bytes = (size_t)(s->T + 1) * 32 * sizeof(float);
    if (dy && acc_bytes <= 200 * 1024) {
        cudaError_t e = acc_bytes > 48 * 1024 ? smem_at_least((const void *)seed_grads_dy_kernel, acc_bytes) : cudaSuccess;
        if (e) return e;
        seed_grads_dy_kernel<<<dim3(s->B, ceil_div(s->H, 32)), 32, acc_bytes, s->stream>>>(s->T, s->B, s->H, top,
                                                                                           d_top_h, dy, s->dhist_h);
        s->launches += 1;
        return cudaGetLastError();
    }
    const size_t n = (size_t)s->B * s->H;
    const unsigned grid = (unsigned)std::min<size_t>(ceil_div(n, 256), (size_t)s->num_sms * 16);
    // the (virtual, in push-only mode) history index of the top at each real time
    seed_grads_kernel<<<grid, 256, 0, s->stream>>>(s->T, s->B, s->H, top, d_top_h, dy, s->dhist_h);
    s->launches += 1;
    return cudaGetLastError();
}

// ------------------------------------------------------------ allocation-free prepass
// stacklstm_pointers_noalloc runs the prepass above for callers that cannot allocate
// device memory. Its scratch (the slot-tag stack, the last-writer table and a status
// word) is this file-scope array, which every GPU that loads the library holds until
// the process exits. Every call shares it and it keeps the last call's contents.
namespace {
constexpr size_t kNoAllocMaxSlots = (size_t)1 << 20;  // (T + 1) * B at most
constexpr int kNoAllocMaxDevices = 64;
__device__ __align__(256) int32_t g_noalloc_scratch[2 * kNoAllocMaxSlots + 64];

std::mutex g_noalloc_mu;
int32_t *g_noalloc_addr[kNoAllocMaxDevices] = {};

// Device address of the scratch on the current device (the host-side name of the array
// is only a stand-in). Looked up once per device.
cudaError_t noalloc_scratch(int32_t **out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kNoAllocMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_addr[dev]) {
        void *p = nullptr;
        if ((e = cudaGetSymbolAddress(&p, g_noalloc_scratch)) != cudaSuccess) return e;
        g_noalloc_addr[dev] = (int32_t *)p;
    }
    *out = g_noalloc_addr[dev];
    return cudaSuccess;
}
}  // namespace
}  // namespace sl

extern "C" sl_status stacklstm_pointers_noalloc(int T, int B, const int8_t *ops, int32_t *p_traj, int32_t *src,
                                                void *stream)
{
    using namespace sl;
    if (T < 1 || B < 1 || !ops || !p_traj || !src) return SL_ERR_ARG;
    if ((size_t)(T + 1) * (size_t)B > kNoAllocMaxSlots) return SL_ERR_UNSUPPORTED;
    cudaStream_t st = (cudaStream_t)stream;
    int32_t *scratch = nullptr;
    if (noalloc_scratch(&scratch) != cudaSuccess) {
        cudaGetLastError();
        return SL_ERR_CUDA;
    }
    int32_t *tags = scratch, *last = scratch + kNoAllocMaxSlots, *err = scratch + 2 * kNoAllocMaxSlots;
    // the status word must start at zero; the kernel initialises every slot tag it reads
    if (cudaMemsetAsync(err, 0, sizeof(int32_t), st) != cudaSuccess) {
        cudaGetLastError();
        return SL_ERR_CUDA;
    }
    prepass_kernel<<<ceil_div(B, kPrepassThreads), kPrepassThreads, 0, st>>>(T, B, ops, p_traj, src, last, tags, err);
    int32_t h = 0;
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess) e = cudaMemcpyAsync(&h, err, sizeof h, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return SL_ERR_CUDA;
    }
    return (sl_status)h;
}

