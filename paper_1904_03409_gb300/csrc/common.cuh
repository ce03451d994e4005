// common.cuh -- internal declarations shared by the library's translation units.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <vector>

#include "../../include/stacklstm.h"

// Most handles one grouped call (stacklstm_forward_group / _backward_group) takes.
constexpr int kMaxGroup = 4;

// A planned persistent step kernel: one cooperative launch runs all T steps.
struct PersistPlan {
    int on = 0;         // 1: persistent; 0: one launch per step
    int U = 0;          // hidden units per column tile
    int EP = 1;         // epilogue warps per tensor-memory lane quadrant (4 * EP epilogue warps)
    int G = 1;          // contraction chunks per ring stage
    int S = 0;          // ring stages
    int slot = 0;       // CTAs per column tile (each takes every slot-th row tile)
    int w_res = 0;      // weight tile resident in shared memory
    int cl = 1;         // thread-block cluster size (the one-row-tile cluster kernels; the KS parts
                        // of a split contraction; 1 otherwise)
    int KS = 1;         // contraction parts per column tile (backward split contraction)
    int n_ct = 0;       // column tiles, padded to a multiple of cl
    unsigned smem = 0;  // dynamic shared memory per CTA
    int threads = 0;    // threads per CTA
    int per_sm = 1;     // co-resident CTAs per SM at this footprint
    int n_dx = 0;       // backward: extra CTAs computing dx on the SMs the steps leave idle
    int dx_S = 0;       // their ring stages
};

// The handle: problem sizes, stream, and the device workspace it owns.
struct stacklstm {
    int T = 0, B = 0, I = 0, H = 0;
    sl_dtype dt = SL_FP32;
    int device = 0;
    cudaStream_t stream = nullptr;
    // the gradient history is cleared on a side stream during the forward: `side_go` marks
    // the caller's stream before the forward steps, `cleared` the end of the clearing
    cudaStream_t side = nullptr;
    cudaEvent_t side_go = nullptr, cleared = nullptr;
    cudaEvent_t join = nullptr;  // grouped calls: marks this handle's stream for the others
    // work overlapped on the side stream (the forward setup beside the prepass, dx beside
    // dW): `aux_go` marks the caller's stream before it, `aux_done` its end
    cudaEvent_t aux_go = nullptr, aux_done = nullptr;
    int clear_queued = 0;
    int async = 0;
    int fwd_done = 0;
    int num_sms = 0;
    int prepass_smem = 0;  // dynamic shared memory of the index prepass (0: global scratch)
    int walk_push_smem = 0;      // the same for the push-only walk (slot tags and index map; 0: separate kernels)
    int walk_built_virtual = 0;  // the last prepass also built the push-only timeline
    int fp32_one_cta = 0;        // fp32: every step of each direction in one CTA (small B * H)
    int pfinal_written = 0;      // the last prepass also wrote the caller's final pointers

    // integer bookkeeping, written by the prepass (all [T+1][B] int32)
    int32_t *p_traj = nullptr;     // pointer before step t (t = T: after the last step)
    int32_t *top = nullptr;        // history index of the top at time t ("src")
    int32_t *slot_last = nullptr;  // history index last written to each slot (-1: never)
    int32_t *slot_scratch = nullptr;  // global slot-tag stack when it does not fit on chip
    int32_t *err = nullptr;           // device-detected status (first error wins)

    // push-only mode (stacklstm_set_mode): the step kernels run over a virtual timeline
    // in which virtual step k of instance b is its k-th push; only push steps' writes are
    // ever read (Sec. 3, Observation 2), so the other steps need no computation
    int push_only = 0;
    int Tr = 0;                  // steps the step kernels run: T, or the most pushes of any instance
    int32_t *vtop = nullptr;     // [T+1][B] virtual history index each virtual step reads
    int32_t *vmap = nullptr;     // [T+1][B] real history index -> virtual index (-1: a non-push write)
    int32_t *vy = nullptr;       // [T+1][B] vmap[top[t][b]]: virtual index of the top at real time t
    int32_t *vslot = nullptr;    // [T+1][B] virtual index of the state last pushed into each slot (-1: none)
    int32_t *xidx = nullptr;     // [T][B] real step of virtual step k (-1: past the instance's pushes)
    int32_t *vstep = nullptr;    // [T][B] virtual step of real step t (-1: not a push)
    void *x_push = nullptr;      // [T][B][I] bf16: x of each virtual step (zero past the pushes)
    int32_t *kmax = nullptr;     // device: the most pushes of any instance
    int32_t *kmax_host = nullptr;  // pinned host copy

    // forward state, write-once history: index 0 = initial state, t+1 = written at step t
    void *hist_h = nullptr;  // [T+1][B][H] dtype
    void *hr = nullptr;      // bf16: [T+1][B][H] h operand of each step, hr[t][b] = hist_h[top[t][b]][b]
    float *hist_c = nullptr;  // [T+1][B][H]
    void *gates = nullptr;    // [T][B][4H] activated i,f,g,o (fp32 path: float, bf16: half)
    void *a_rm = nullptr;     // [T][B][I+H] the contraction operand [x_t ; h_read] (dtype)

    // backward state
    float *dhist_h = nullptr;  // [T+1][B][H] gradient w.r.t. each history state
    float *dhist_c = nullptr;  // [T+1][B][H]
    void *dG = nullptr;        // [T][B][4H] gate pre-activation gradients (fp32 / bf16)

    // packed weights (taken at forward)
    void *w_fwd = nullptr;  // fp32: W^T [4H][I+H] float; bf16: forward operand tiles
    void *w_bwd = nullptr;  // bf16: backward operand tiles
    void *w_dx = nullptr;   // bf16: input-gradient operand tiles
    float *dw_part = nullptr;  // split-K partials of the weight-gradient contraction
    size_t dw_part_elems = 0;
    const void *x_saved = nullptr;  // the caller's x, read again by the weight gradient

    // bf16 tensor-core plan (bf16_path.cu)
    int uf = 0, ub = 0;      // hidden units per CTA tile: forward, backward
    int kcx = 0, kcf = 0, kcb = 0;  // 64-wide contraction chunks: x part, forward total, backward
    int sf = 0, sb = 0, sx = 0, sw = 0;  // ring depths: forward, backward, dx, dW
    alignas(64) unsigned char tmaps[10][128] = {};  // TMA descriptors (bf16_path.cu)
    // persistent step kernels (one launch for all T steps; bf16_persist.cu)
    PersistPlan pf, pb;            // forward, backward (on = 0: one launch per step)
    PersistPlan fc;                // forward as one thread-block cluster (one row tile; bf16_cluster.cu)
    void *g_fcl = nullptr;         // its h slice blocks [T][column tiles][2 KB]
    PersistPlan bc;                // backward as one thread-block cluster (one row tile; bf16_cluster.cu)
    PersistPlan cc;                // small batches: both directions on CUDA cores (bf16_small.cu)
    void *w_ccf = nullptr, *w_ccb = nullptr;  // their weight slices
    void *w_bcl = nullptr;         // its weight chunks
    void *g_bcl = nullptr;         // its swizzled dG blocks [T][column tiles][8 KB]
    int32_t *rowcnt = nullptr;     // [2][row tiles][cnt_stride] completed steps per row tile
    int cnt_stride = 32;           // ints between two row tiles' counters (one 128-byte line each)
    float *split_part = nullptr;   // backward split contraction: partial dh_read rows
    int32_t *split_cnt = nullptr;  // backward split contraction: partials written per tile pair
    int nx = 0, nxt = 0;     // input gradient: columns per tile, number of column tiles
    int dw_mt = 0, dw_nt = 0, dw_split = 0;  // weight gradient: m tiles, column tiles, splits
    int dw_ntile = 0;                        // weight gradient: gate columns per tile
    int dw_mtile = 0;                        // weight gradient: m rows per tile (128 or 256)
    long long wait_limit = 0;  // clock cycles one bounded device-side wait may spin
    long long wait_limit_bwd = 0;  // the same for the backward's kernels (its own test hook)

    // launch accounting and optional per-phase event timing (api.cu)
    long long launches = 0;  // kernel launches of this library, running total
    int timing = 0;
    int cur_phase = -1;
    double phase_ms[SL_NUM_PHASES] = {};
    long long phase_launches[SL_NUM_PHASES] = {};
    struct EventPair {
        int phase;
        cudaEvent_t a, b;
    };
    std::vector<EventPair> pending;
    std::vector<cudaEvent_t> event_pool;

    std::string plan;  // stacklstm_plan
    std::string last_error;
    std::vector<void *> allocs;
};

namespace sl {

// ---- index / gather kernels (index_kernels.cu)
// also writes the final pointers to p_final (if given) when the walk runs on chip
// (s->pfinal_written)
cudaError_t launch_prepass(stacklstm *s, const int8_t *ops, int32_t *p_final);
// Raise kernel `fn`'s dynamic shared-memory limit on the current device to at least
// `bytes`. The limit belongs to the function, not to a handle, so handles of different
// sizes (created in any order, used from any stream) only ever raise it.
cudaError_t smem_at_least(const void *fn, size_t bytes);
cudaError_t launch_gather_rows(stacklstm *s, const int32_t *idx, int rows, size_t elem_bytes,
                               const void *hist, void *out, int row_elems);
cudaError_t launch_seed_grads(stacklstm *s, const float *d_top_h, const float *dy);
// push-only mode: the virtual timeline's indices from the prepass's (kernel), and the
// number of virtual steps (read back to the host: synchronizes the stream)
cudaError_t launch_compact(stacklstm *s);
cudaError_t read_virtual_steps(stacklstm *s);
// push-only mode: zero the rows of dx [T][B][I] that belong to non-push steps
cudaError_t launch_zero_nonpush_rows(stacklstm *s, float *dx);

// ---- fp32 CUDA-core path (fp32_path.cu)
// plans the fp32 path (s->fp32_one_cta) and describes it
std::string fp32_describe(stacklstm *s);
cudaError_t fp32_forward_setup(stacklstm *s, const float *h0, const float *c0, const float *W);
cudaError_t fp32_forward_steps(stacklstm *s, const float *x, const float *W, const float *bias);
cudaError_t fp32_backward_steps(stacklstm *s);
cudaError_t fp32_dx(stacklstm *s, float *dx);
cudaError_t fp32_dw(stacklstm *s, float *dW, float *dbias);

// ---- bf16 tensor-core path (bf16_path.cu)
cudaError_t bf16_prepare(stacklstm *s);
// the forward's inputs: the virtual steps' x gathered (push-only mode), the x tensor maps
cudaError_t bf16_forward_setup_x(stacklstm *s, const __nv_bfloat16 *x);
// the initial state into history row 0, the weight tiles packed (needs no index)
cudaError_t bf16_forward_setup_state(stacklstm *s, const __nv_bfloat16 *h0, const float *c0, const __nv_bfloat16 *W);
cudaError_t bf16_forward_steps(stacklstm *s, const float *bias);
// the last step's pointwise backward; with d_top_h it also seeds the final tops' gradients
// (the caller seeds them itself when the loss also has per-step terms)
cudaError_t bf16_backward_setup(stacklstm *s, const float *d_top_h);
cudaError_t bf16_backward_steps(stacklstm *s, float *dx, bool *dx_done);
// Grouped calls: true when the n handles' step kernels can run as one launch (every one
// on the one-row-tile cluster kernels of the same cluster size); that launch, on `st`.
bool bf16_can_group(stacklstm *const *hs, int n, bool fwd);
cudaError_t bf16_forward_steps_group(stacklstm *const *hs, int n, const float *const *bias, cudaStream_t st);
cudaError_t bf16_backward_steps_group(stacklstm *const *hs, int n, cudaStream_t st);
cudaError_t bf16_dx(stacklstm *s, float *dx);
cudaError_t bf16_dw(stacklstm *s, float *dW, float *dbias);
// push-only mode: x of each virtual step into s->x_push (bf16 rows)
cudaError_t bf16_gather_push_x(stacklstm *s, const __nv_bfloat16 *x);
size_t bf16_workspace_bytes(int T, int B, int I, int H, int num_sms);
const char *bf16_unsupported(int T, int B, int I, int H);
std::string bf16_describe(const stacklstm *s);

// generic tensor-core contraction (bf16_path.cu): D [splits][R][N] fp32 = A [R][K] B^T,
// A bf16 row-major (rows lda apart), B packed by bf16_pack_kmajor from src (rows n of
// length K, or with trans the columns of a [K][N] src)
size_t bf16_kmajor_bytes(int N, int K);
cudaError_t bf16_pack_kmajor(const __nv_bfloat16 *src, size_t ld, bool trans, int N, int K, void *out,
                             cudaStream_t st, int num_sms);
cudaError_t bf16_gemm(const __nv_bfloat16 *A, size_t lda, int R, int K, const void *bpack, int N, float *D, int splits,
                      cudaStream_t st, int num_sms, long long limit, int32_t *err);

inline unsigned ceil_div(size_t a, size_t b) { return (unsigned)((a + b - 1) / b); }

}  // namespace sl
