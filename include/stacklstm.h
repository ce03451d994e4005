/*
 * stacklstm.h -- C ABI of the GB300 (sm_103a) homogenized StackLSTM step.
 *
 * The library runs the minibatched, homogenized StackLSTM of Ding & Koehn,
 * "Parallelizable Stack Long Short-Term Memory" (arXiv:1904.03409), forward and
 * backward, on one GPU:
 *   - every step, every instance b reads the (h, c) state at its stack-top pointer p[b],
 *     computes the LSTM gates from [x_t ; h_p] with one fused gate contraction, writes
 *     the new state to stack slot p[b] + 1 and moves p[b] by its op (push +1, pop -1,
 *     hold 0), whatever the op is (Algorithm 1; unified pointer update, Sec. 3);
 *   - the step output is the top after the pointer update (Algorithm 1, return value);
 *   - cell states move with hidden states (footnote to Sec. 2);
 *   - the backward runs in reverse time and routes gradients to every state a step read,
 *     including states later popped or overwritten (Sec. 5).
 *
 * LSTM cell (the paper names only "LSTM"): z = [x ; h] W + bias with W of shape
 * [I + H, 4H], row-major, gate column blocks in the order i, f, g, o;
 * i, f, o = sigmoid, g = tanh; c' = f c + i g; h' = o tanh(c').
 *
 * Conventions for every call below:
 *   - All tensor pointers are DEVICE pointers on the handle's device, C-ordered
 *     (row-major, last index fastest), owned by the caller, and must be 16-byte aligned.
 *   - Calls are asynchronous with respect to the GPU and ordered on the handle's stream.
 *     In the default synchronous mode, forward and backward synchronize the stream before
 *     returning and report device-detected errors (bad op, underflow); in async mode
 *     (stacklstm_set_async) they return after enqueueing and stacklstm_status reports.
 *   - No call aborts, traps or prints. Each returns a status; stacklstm_last_error gives
 *     a one-line message for the last failure on a handle.
 *   - Device-detected errors never cause out-of-bounds accesses: a bad op or a pop at
 *     depth 0 is recorded and then treated as a hold, so every index stays in range.
 *
 * Element types by dtype:
 *   SL_FP32: x, h0, W, h_stack, y are float; every computation in fp32 on CUDA cores
 *            (no tensor cores, no TF32).
 *   SL_BF16: x, h0, W, h_stack, y are bf16 (uint16 bit patterns); the gate contractions
 *            run on tcgen05 tensor cores with fp32 accumulation; cell states, gradients
 *            and all accumulations are fp32. Requires I % 8 == 0 and H % 8 == 0.
 *   c0, c_stack, bias and every gradient are float in both modes.
 */
/*
 * Test hooks. stacklstm_create reads these environment variables; they exist so that the
 * tests can reach every kernel plan the library has on shapes where the planner would pick
 * another one. Results are the same under every setting (within the stated tolerances);
 * only speed changes. Unset, the planner decides.
 *   STACKLSTM_WAIT_LIMIT_CYCLES=n  clock budget of one bounded device-side wait
 *                                  (default 4e9); 0 makes every wait run out at once, so
 *                                  calls report SL_ERR_TIMEOUT
 *   STACKLSTM_WAIT_LIMIT_BWD_CYCLES=n  the same budget for the backward's kernels only
 *                                  (default: STACKLSTM_WAIT_LIMIT_CYCLES), so that a
 *                                  forward can complete before the backward times out
 *   STACKLSTM_STEP_KERNELS=1       one launch per time step instead of the persistent and
 *                                  cluster kernels (fp32: instead of one CTA for all steps)
 *   STACKLSTM_FWD_CLUSTER=0        no thread-block-cluster forward for one row tile
 *   STACKLSTM_BWD_CLUSTER=0        no thread-block-cluster backward for one row tile
 *   STACKLSTM_BWD_SPLIT=k          the persistent backward with its 4H contraction split
 *                                  over k CTAs per 64-unit column tile (k = 4)
 *   STACKLSTM_SPLIT_CLUSTER=0      the parts of a split contraction trade their partial
 *                                  sums through an L2 scratch, not as a thread-block
 *                                  cluster in shared memory
 *   STACKLSTM_DX_SPARE=0 | k       dx in its own launch (0), or by at most k extra CTAs of
 *                                  the persistent backward launch (whole clusters of it,
 *                                  when that launch is a cluster launch)
 *   STACKLSTM_DW_M=128 | 256       the weight gradient's tile: 128 or 256 rows of W (x 256
 *                                  gate columns) per CTA
 *   STACKLSTM_CUDA_CORE=0 | 1      small batches (B <= 32, H <= 256): never (0), or
 *                                  whenever the shape allows (1), the CUDA-core cluster
 *                                  kernels instead of the tensor-core ones
 */
#ifndef STACKLSTM_H
#define STACKLSTM_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct stacklstm *stacklstm_t;

typedef enum {
    SL_OK = 0,
    SL_ERR_ARG = 1,         /* null handle or pointer, size out of range, misaligned pointer */
    SL_ERR_OP = 2,          /* an op outside {-1, 0, +1} (the op set of Sec. 3)            */
    SL_ERR_UNDERFLOW = 3,   /* a pop at stack depth 0 (undefined in the paper)             */
    SL_ERR_STATE = 4,       /* backward without a completed forward on the handle          */
    SL_ERR_CUDA = 5,        /* a CUDA runtime error (message in stacklstm_last_error)       */
    SL_ERR_TIMEOUT = 6,     /* a bounded device-side wait ran out; the context stays usable */
    SL_ERR_UNSUPPORTED = 7, /* sizes or device this build's kernels do not support         */
    SL_ERR_OOM = 8          /* device workspace allocation failed                          */
} sl_status;

typedef enum { SL_FP32 = 0, SL_BF16 = 1 } sl_dtype;

/*
 * stacklstm_create -- allocate a handle and its device workspace for one problem size.
 *   T      time steps (>= 1); the stack has T + 1 slots, so it can never overflow
 *          (the paper fixes 150 slots, Sec. 4.1; here capacity follows T).
 *   B      batch instances (>= 1); I input width (>= 1); H hidden width (>= 1).
 *   dtype  SL_FP32 or SL_BF16 (see above).
 *   device CUDA device ordinal; stream: a cudaStream_t (NULL = legacy default stream).
 * The workspace (state history, saved gates, gradient history, indices) is owned by the
 * handle until stacklstm_destroy. Returns SL_ERR_ARG, SL_ERR_UNSUPPORTED or SL_ERR_OOM
 * on failure, leaving *out NULL.
 */
sl_status stacklstm_create(stacklstm_t *out, int T, int B, int I, int H, sl_dtype dtype,
                           int device, void *stream);

/* Replace the stream later calls are ordered on. */
sl_status stacklstm_set_stream(stacklstm_t s, void *stream);

/* async != 0: forward/backward return after enqueueing; stacklstm_status reports. */
sl_status stacklstm_set_async(stacklstm_t s, int async);

/*
 * stacklstm_forward -- T homogenized steps (Algorithm 1) for all B instances.
 * Inputs:
 *   x     [T, B, I]  input vectors x_t (dtype)
 *   ops   [T, B]     int8 ops in {-1, 0, +1}; a pop needs depth > 0
 *   h0    [B, H]     initial hidden state, stack slot 0 (dtype)
 *   c0    [B, H]     initial cell state (float)
 *   W     [I+H, 4H]  gate weights (dtype); rows 0..I-1 act on x, rows I.. on h
 *   bias  [4H]       gate bias (float)
 * Outputs (all nullable except p_final):
 *   h_stack [T+1, B, H] final slot-indexed stack, hidden part (dtype); slot 0 is h0,
 *                       slots no step wrote are 0. Slots above the top hold what
 *                       Algorithm 1 last wrote there.
 *   c_stack [T+1, B, H] the same for cell states (float)
 *   p_final [B]         final stack pointers
 *   p_traj  [T+1, B]    pointer before each step and after the last (p_traj[0] = 0);
 *                       step t reads slot p_traj[t] and writes slot p_traj[t] + 1
 *   src     [T+1, B]    provenance of the top at each time: 0 is the initial state,
 *                       t + 1 is the state written at step t; src[t] is what step t read
 *   y       [T, B, H]   step outputs: h at the top after step t's pointer move (dtype)
 * The handle keeps what backward needs (packed copies of W, the state history, the
 * gates), so W may change after forward returns; x must stay valid and unchanged until
 * the matching backward returns (the weight gradient reads it again).
 */
sl_status stacklstm_forward(stacklstm_t s, const void *x, const int8_t *ops, const void *h0,
                            const float *c0, const void *W, const float *bias, void *h_stack,
                            float *c_stack, int32_t *p_final, int32_t *p_traj, int32_t *src,
                            void *y);

/*
 * stacklstm_backward -- reverse-time backward of the last forward on this handle for the
 * loss L = sum(d_top_h * h_top_final) + sum_t sum(dy_t * y_t).
 * Inputs (nullable; NULL means zero): d_top_h [B, H], dy [T, B, H] (float).
 * Outputs (float; each nullable): dx [T, B, I], dh0 [B, H], dc0 [B, H],
 * dW [I+H, 4H], dbias [4H]. Gradients are overwritten, not accumulated.
 * Every reduction runs in a fixed order with no atomics, so results are bitwise
 * reproducible run to run. Returns SL_ERR_STATE without a preceding forward.
 */
sl_status stacklstm_backward(stacklstm_t s, const float *d_top_h, const float *dy, float *dx,
                             float *dh0, float *dc0, float *dW, float *dbias);

/*
 * Modes of the step computation.
 *   SL_MODE_HOMOGENIZED (default): Algorithm 1 as written. Every instance runs the LSTM
 *     cell at every step, whatever its op, and writes slot p + 1.
 *   SL_MODE_PUSH_ONLY: dead writes skipped. By Observation 2 of Sec. 3 a pop or hold step
 *     writes slot p + 1 above the new top, and the next push overwrites that slot before
 *     the pointer reaches it, so only push steps' writes are ever read. This mode runs
 *     the cell for push steps only: virtual step k of instance b is its k-th push, and
 *     the step kernels run max_b(pushes of b) steps instead of T. p_final, p_traj, src,
 *     y and every gradient are those of the homogenized mode (y and dx bit for bit; dW
 *     and dbias are sums in another order). h_stack / c_stack hold the stack of the
 *     push/pop definition of Sec. 2: each slot the state last pushed into it (0 if
 *     none). They equal the homogenized mode's on the live part (slots 0 .. p_final);
 *     above the top, Algorithm 1 leaves what a pop or hold step wrote last, states
 *     nothing reads. bf16 path only.
 *     Its forward synchronizes the handle's stream once, after the index prepass, to
 *     learn the number of virtual steps (also in async mode).
 */
typedef enum { SL_MODE_HOMOGENIZED = 0, SL_MODE_PUSH_ONLY = 1 } sl_mode;

/*
 * stacklstm_set_mode -- choose the mode of later forward calls. Switching modes needs a
 * new forward before backward (SL_ERR_STATE otherwise). The first switch to
 * SL_MODE_PUSH_ONLY allocates its workspace (about (T + 1) B 24 + T B 2 I bytes):
 * SL_ERR_OOM if that fails; SL_ERR_UNSUPPORTED on the fp32 path. Synchronizes the
 * handle's stream.
 */
sl_status stacklstm_set_mode(stacklstm_t s, sl_mode mode);

/* Number of steps the step kernels ran in the last forward: T in the homogenized mode,
 * the most pushes of any instance (at least 1) in the push-only mode. */
sl_status stacklstm_steps_run(stacklstm_t s, int *steps);

/*
 * Grouped calls: the forward (backward) of up to 4 handles on one device in one call. A
 * transition-based parser runs several StackLSTMs over one batch (the stack, the buffer
 * and the action history of Sec. 4.1; Table 1 gives each transition's stack and buffer
 * ops); with the transitions known, their recurrences are independent of one another.
 * The result is that of calling stacklstm_forward (stacklstm_backward) on each handle,
 * each on its own stream. When every handle runs the one-row-tile cluster kernels (B <= 64)
 * with the same cluster size (the same H), their step kernels run as ONE launch of one
 * thread-block cluster per handle, on the first handle's stream; each handle's stream
 * joins that stream before the launch and waits for it afterwards. Otherwise each handle
 * launches its own. The work before and after the steps stays on each handle's stream.
 * Timing: the one launch counts in the first handle's forward (backward) phase.
 * Returns the first failing handle's status (SL_ERR_ARG: n outside 1..4, a null or
 * repeated handle, handles on different devices).
 */
typedef struct {
    const void *x;        /* as stacklstm_forward's arguments of the same names */
    const int8_t *ops;
    const void *h0;
    const float *c0;
    const void *W;
    const float *bias;
    void *h_stack;
    float *c_stack;
    int32_t *p_final;
    int32_t *p_traj;
    int32_t *src;
    void *y;
} sl_forward_args;

typedef struct {
    const float *d_top_h;  /* as stacklstm_backward's arguments of the same names */
    const float *dy;
    float *dx;
    float *dh0;
    float *dc0;
    float *dW;
    float *dbias;
} sl_backward_args;

sl_status stacklstm_forward_group(int n, const stacklstm_t *hs, const sl_forward_args *args);
sl_status stacklstm_backward_group(int n, const stacklstm_t *hs, const sl_backward_args *args);

/*
 * Phases of a forward + backward, as stacklstm_get_timing reports them. Each phase is a
 * contiguous run of kernel launches on the handle's stream.
 */
typedef enum {
    SL_PHASE_PREPASS = 0,    /* op validation and the index prepass                              */
    SL_PHASE_FORWARD = 1,    /* the forward steps (one persistent launch, or T launches)         */
    SL_PHASE_OUTPUTS = 2,    /* optional forward outputs (y, h_stack, c_stack, p_traj)           */
    SL_PHASE_BACKWARD = 3,   /* the reverse-time backward steps (one launch, or T / 2T launches) */
    SL_PHASE_DX = 4,         /* the input-gradient contraction dx = dG W_x^T                     */
    SL_PHASE_DW = 5,         /* the weight- and bias-gradient contraction and its reduction      */
    SL_PHASE_FWD_SETUP = 6,  /* weight packing and the initial state, before the forward steps   */
    SL_PHASE_BWD_SETUP = 7,  /* clearing and seeding the gradient history, last-step pointwise   */
    SL_NUM_PHASES = 8
} sl_phase;

/*
 * stacklstm_set_timing -- on != 0: record a CUDA event pair on the handle's stream around
 * every phase of later calls. Resets the accumulated times and launch counts either way.
 */
sl_status stacklstm_set_timing(stacklstm_t s, int on);

/*
 * stacklstm_get_timing -- synchronize the handle's stream and write, for the first n
 * phases (n <= SL_NUM_PHASES), the device time in milliseconds accumulated since the last
 * stacklstm_set_timing (ms, nullable; zeros for phases run while timing was off) and the
 * number of this library's kernel launches (launches, nullable; always counted).
 * Host pointers.
 */
sl_status stacklstm_get_timing(stacklstm_t s, double *ms, long long *launches, int n);

/* Synchronize the handle's stream and return (then clear) any device-detected error. */
sl_status stacklstm_status(stacklstm_t s);

/* Free the handle and its workspace (synchronizes its stream first). NULL is a no-op. */
sl_status stacklstm_destroy(stacklstm_t s);

/* Static, human-readable name of a status code. */
const char *stacklstm_status_string(sl_status st);

/* One-line description of how the handle runs: dtype path, kernels (persistent or one
 * launch per step), tile sizes, cluster sizes, ring depths. Valid until the handle is
 * destroyed. */
const char *stacklstm_plan(stacklstm_t s);

/* One-line message for the last failure on the handle ("" if none). Valid until the
 * next call on the handle. */
const char *stacklstm_last_error(stacklstm_t s);

/*
 * stacklstm_pointers_noalloc -- the index prepass alone (pointer trajectory and read
 * provenance of every instance), for callers that cannot allocate device memory when
 * they need it: services whose device memory is all reserved up front by a pooling
 * allocator (a library's own cudaMalloc then fails, or takes memory the pool counted
 * on), and callers that must not let a cudaMalloc or cudaFree synchronize the device
 * while other streams are busy. It needs no handle and allocates nothing: it calls no
 * cudaMalloc, cudaFree or allocating routine.
 * The paper has no counterpart; it is a convenience of this library.
 *   T, B     sizes; (T + 1) * B must not exceed 1,048,576, else SL_ERR_UNSUPPORTED
 *   ops      [T, B] int8 device pointer, ops in {-1, 0, +1}
 *   p_traj   [T + 1, B] int32 device output, as stacklstm_forward's p_traj
 *   src      [T + 1, B] int32 device output, as stacklstm_forward's src
 *   stream   cudaStream_t (NULL = legacy default stream)
 * The three pointers must belong to the current device, which runs the kernel. The call
 * enqueues the prepass on `stream`, then reads its status word back to the host and
 * synchronizes `stream` before it returns.
 * Returns SL_OK, SL_ERR_OP / SL_ERR_UNDERFLOW (bad op stream; indices are still written,
 * bad ops run as holds), SL_ERR_ARG, SL_ERR_UNSUPPORTED or SL_ERR_CUDA.
 * Scratch: an 8 MiB array in the library's device memory, held on every GPU that loads
 * the library until the process exits. All calls share it, so calls that overlap on a
 * GPU (other streams, other host threads) race; it keeps the previous call's contents
 * and the call itself clears what must start at zero. The first call on a device looks
 * up the array's device address (a one-time set-up on that device).
 */
sl_status stacklstm_pointers_noalloc(int T, int B, const int8_t *ops, int32_t *p_traj, int32_t *src,
                                     void *stream);

/*
 * The parser head after the three StackLSTMs of a transition-based parser: the stack,
 * the buffer and the action history (Sec. 4.1, which uses arc-hybrid; Table 1 gives each
 * transition's stack and buffer ops). Before transition k of instance b the head reads
 * the three tops (the output of Algorithm 1 of each StackLSTM):
 *   s  = y_stack[k - 1, b]          (h0_stack[b] when k = 0)
 *   bu = y_buffer[n[b] - 1 + k, b]  (the buffer StackLSTM is filled by n[b] pushes first)
 *   a  = y_action[k - 1, b]         (h0_action[b] when k = 0)
 * and computes p = ReLU(Wp [s; bu; a] + dp), the parser state (P wide; 200 in Sec. 4.1),
 * z = Wz p + q over the A transitions, and the row loss logsumexp(z) - z[gold[k, b]].
 * Transitions k >= L[b] are padding: no loss, no gradient. The paper fixes only the
 * state width; the ReLU layer and the softmax follow the parser architecture its
 * experiments reuse. bf16 inputs; the contractions U Wp^T, dP Wp and dP^T U over all rows
 * on the tensor cores (bf16 operands, dP rounded to bf16, fp32 accumulation), the rest in
 * fp32; deterministic.
 *
 * stacklstm_head_create -- a head for T transitions (the stack and action StackLSTMs'
 *   step count), a buffer StackLSTM of Tb steps, B instances, hidden width H (a multiple
 *   of 8), state width P (a multiple of 8, <= 256) and A transitions (2..8). Owns its
 *   workspace: about T B (24 H + 8 P + 16) bytes for the gathered tops, the states and the
 *   gradients, plus up to 32 x 3H x P floats of weight-gradient partial sums. Calls are
 *   ordered on `stream`;
 *   SL_ERR_ARG (bad size or device), SL_ERR_UNSUPPORTED or SL_ERR_OOM on failure,
 *   leaving *out NULL.
 */
typedef struct stacklstm_head *stacklstm_head_t;
sl_status stacklstm_head_create(stacklstm_head_t *out, int T, int Tb, int B, int H, int P, int A, int device,
                                void *stream);

/*
 * stacklstm_head_run -- loss and gradients of the head, enqueued on the head's stream.
 * Inputs (device pointers; StackLSTM outputs 16-byte aligned):
 *   y_stack, y_action [T, B, H] bf16; y_buffer [Tb, B, H] bf16; h0_stack, h0_action
 *   [B, H] bf16; n, L [B] int32 (sentence lengths, transitions per instance);
 *   gold [T, B] int8 transition ids in [0, A) for k < L[b]; Wp [P, 3H] bf16; dp [P];
 *   Wz [A, P]; q [A] (float).
 * Outputs (float, device):
 *   loss_rows [T, B] (0 on padding; the loss is their sum);
 *   dy_stack, dy_action [T, B, H] and dy_buffer [Tb, B, H]: the gradient of the loss
 *     w.r.t. each StackLSTM output, to pass as stacklstm_backward's dy (rows the head
 *     does not read are 0);
 *   dWp [P, 3H], ddp [P], dWz [A, P], dq [A].
 * The gradients w.r.t. h0_stack and h0_action (the k = 0 reads) stay in the workspace
 * for stacklstm_head_add_h0_grads. A transition whose length or label is out of range is
 * skipped and reported by stacklstm_head_status (SL_ERR_ARG).
 */
sl_status stacklstm_head_run(stacklstm_head_t h, const void *y_stack, const void *h0_stack, const void *y_buffer,
                             const void *y_action, const void *h0_action, const int32_t *n, const int32_t *L,
                             const int8_t *gold, const void *Wp, const float *dp, const float *Wz, const float *q,
                             float *loss_rows, float *dy_stack, float *dy_buffer, float *dy_action, float *dWp,
                             float *ddp, float *dWz, float *dq);

/* Add the last run's gradients w.r.t. h0_stack and h0_action into dh0_stack and
 * dh0_action ([B, H] float, device; either may be NULL): call it after the StackLSTMs'
 * stacklstm_backward wrote their dh0, to get the whole gradient of the initial states. */
sl_status stacklstm_head_add_h0_grads(stacklstm_head_t h, float *dh0_stack, float *dh0_action);

/* Synchronize the head's stream; return (then clear) a device-detected error. */
sl_status stacklstm_head_status(stacklstm_head_t h);

/* Free the head and its workspace (synchronizes its stream first). NULL is a no-op. */
sl_status stacklstm_head_destroy(stacklstm_head_t h);

/* One-line message for the last failure on the head ("" if none). */
const char *stacklstm_head_last_error(stacklstm_head_t h);

#ifdef __cplusplus
}
#endif

#endif /* STACKLSTM_H */
