/*
 * stacklstm_oracle.c -- plain, slow, fp64 CPU oracle of the StackLSTM time step.
 *
 * TEST INFRASTRUCTURE ONLY. Nothing in the product library links, loads or calls this
 * file; only the test suite, the smoke check and the benchmark's CPU-baseline leg do.
 * It shares no code, header, table or helper with the CUDA path.
 *
 * What it computes (Ding & Koehn, "Parallelizable Stack Long Short-Term Memory"):
 *   - One instance at a time, with an explicit stack of (h, c) slots. Slot 0 holds the
 *     initial state; the stack pointer p starts at 0. Cell states travel with hidden
 *     states (footnote to Sec. 2).
 *   - ORACLE_DEFINITION: the original operations of Sec. 2. Push reads slot p, runs the
 *     LSTM on (x_t, h_p), writes slot p+1 and sets p <- p+1; pop sets p <- p-1; hold
 *     (Sec. 3, last paragraph) does nothing.
 *   - ORACLE_HOMOGENIZED: Algorithm 1 taken literally. Every step reads slot p, runs the
 *     LSTM, writes slot p+1, then moves p <- p + op (Sec. 3, unified pointer update),
 *     whatever op is.
 *   - The step output is the top after the pointer update (Algorithm 1, return value).
 *   - LSTM (the paper says only "LSTM"; standard cell, no peepholes, one fused weight):
 *       z = x W[0:I] + h W[I:I+H] + bias, gate column blocks i, f, g, o;
 *       i, f, o = sigmoid, g = tanh, c' = f c + i g, h' = o tanh(c').
 *   - Backward (Sec. 5: gradients reach overwritten, popped states; every intermediate
 *     top is stored once): reverse time over a per-slot gradient stack. At step t, add
 *     dy_t to the slot that is top after the step, take (and clear) the gradient of the
 *     slot written at the step, back-propagate through the cell, and add the gradient
 *     of the state read to the slot that was read. In definition mode only pushes
 *     back-propagate.
 *   - Loss: L = sum(d_top_h * h_top_final) + sum_t sum(dy_t * y_t).
 *
 * Outputs per instance: the pointer trajectory, the provenance ("history index") of the
 * top at every time (0 = the initial state, t+1 = the state written at step t), the
 * step outputs y, the final slot-indexed stack (slots never written read as 0), and the
 * gradients dx, dh0, dc0; dW and dbias are summed over instances in instance order.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum { ORACLE_HOMOGENIZED = 0, ORACLE_DEFINITION = 1 };
enum { ORACLE_OK = 0, ORACLE_BAD_OP = 1, ORACLE_UNDERFLOW = 2, ORACLE_NOMEM = 3, ORACLE_BAD_ARG = 4 };

static double sigm(double z) { return 1.0 / (1.0 + exp(-z)); }

/* Everything one instance needs; pointers into the caller's batched arrays use stride B. */
typedef struct {
    int T, B, I, H, mode, b;
    const double *x, *h0, *c0, *W, *bias, *d_top_h, *dy;
    const int8_t *ops;
    int32_t *p_traj, *src;
    double *y, *stack_h, *stack_c, *dx, *dh0, *dc0;
    double *dW, *dbias; /* the calling thread's partial sums, accumulated into */
} inst_args;

static int run_instance(const inst_args *a)
{
    const int T = a->T, B = a->B, I = a->I, H = a->H, b = a->b;
    const int K = I + H, G = 4 * H, S = T + 1;
    int rc = ORACLE_OK;

    /* explicit stack: S slots of (h, c) plus the provenance tag of each slot */
    double *sh = calloc((size_t)S * H, sizeof(double));
    double *sc = calloc((size_t)S * H, sizeof(double));
    int32_t *tag = calloc((size_t)S, sizeof(int32_t));
    int32_t *written = calloc((size_t)S, sizeof(int32_t));
    int32_t *p = calloc((size_t)S, sizeof(int32_t));
    /* forward tape: per step, the state read and the cell's intermediate values */
    double *t_hr = calloc((size_t)T * H, sizeof(double));
    double *t_cr = calloc((size_t)T * H, sizeof(double));
    double *t_gate = calloc((size_t)T * G, sizeof(double)); /* activated i, f, g, o */
    double *t_cn = calloc((size_t)T * H, sizeof(double));
    int32_t *did = calloc((size_t)(T > 0 ? T : 1), sizeof(int32_t)); /* step ran the cell */
    double *z = calloc((size_t)G, sizeof(double));
    double *ds_h = calloc((size_t)S * H, sizeof(double));
    double *ds_c = calloc((size_t)S * H, sizeof(double));
    double *dz = calloc((size_t)G, sizeof(double));
    if (!sh || !sc || !tag || !written || !p || !t_hr || !t_cr || !t_gate || !t_cn || !did ||
        !z || !ds_h || !ds_c || !dz) {
        rc = ORACLE_NOMEM;
        goto done;
    }

    /* slot 0 = initial state */
    for (int j = 0; j < H; ++j) {
        sh[j] = a->h0[(size_t)b * H + j];
        sc[j] = a->c0[(size_t)b * H + j];
    }
    tag[0] = 0;
    written[0] = 1;
    p[0] = 0;

    /* ---------------- forward ---------------- */
    for (int t = 0; t < T; ++t) {
        const int op = a->ops[(size_t)t * B + b];
        const int pt = p[t];
        if (op != 1 && op != 0 && op != -1) { rc = ORACLE_BAD_OP; goto done; }
        if (pt + op < 0) { rc = ORACLE_UNDERFLOW; goto done; }
        if (a->src) a->src[(size_t)t * B + b] = tag[pt];

        const int runs_cell = (a->mode == ORACLE_HOMOGENIZED) || (op == 1);
        did[t] = runs_cell;
        if (runs_cell) {
            const double *xt = a->x + ((size_t)t * B + b) * I;
            const double *hr = sh + (size_t)pt * H, *cr = sc + (size_t)pt * H;
            /* z = [x_t ; h_read] W + bias */
            for (int n = 0; n < G; ++n) z[n] = a->bias[n];
            for (int k = 0; k < I; ++k) {
                const double ak = xt[k];
                const double *Wk = a->W + (size_t)k * G;
                for (int n = 0; n < G; ++n) z[n] += ak * Wk[n];
            }
            for (int k = 0; k < H; ++k) {
                const double ak = hr[k];
                const double *Wk = a->W + (size_t)(I + k) * G;
                for (int n = 0; n < G; ++n) z[n] += ak * Wk[n];
            }
            double *gt = t_gate + (size_t)t * G;
            for (int j = 0; j < H; ++j) {
                const double ig = sigm(z[j]), fg = sigm(z[H + j]);
                const double gg = tanh(z[2 * H + j]), og = sigm(z[3 * H + j]);
                const double cn = fg * cr[j] + ig * gg;
                gt[j] = ig; gt[H + j] = fg; gt[2 * H + j] = gg; gt[3 * H + j] = og;
                t_hr[(size_t)t * H + j] = hr[j];
                t_cr[(size_t)t * H + j] = cr[j];
                t_cn[(size_t)t * H + j] = cn;
            }
            /* write slot p+1 (after the reads above: slot p+1 != slot p) */
            double *wh = sh + (size_t)(pt + 1) * H, *wc = sc + (size_t)(pt + 1) * H;
            for (int j = 0; j < H; ++j) {
                wc[j] = t_cn[(size_t)t * H + j];
                wh[j] = gt[3 * H + j] * tanh(wc[j]);
            }
            tag[pt + 1] = t + 1;
            written[pt + 1] = 1;
        }
        p[t + 1] = pt + op;
        if (a->y) {
            const double *top = sh + (size_t)p[t + 1] * H;
            for (int j = 0; j < H; ++j) a->y[((size_t)t * B + b) * H + j] = top[j];
        }
    }
    for (int t = 0; t <= T; ++t)
        if (a->p_traj) a->p_traj[(size_t)t * B + b] = p[t];
    if (a->src) a->src[(size_t)T * B + b] = tag[p[T]];
    if (a->stack_h || a->stack_c)
        for (int s = 0; s < S; ++s)
            for (int j = 0; j < H; ++j) {
                const size_t o = ((size_t)s * B + b) * H + j;
                if (a->stack_h) a->stack_h[o] = written[s] ? sh[(size_t)s * H + j] : 0.0;
                if (a->stack_c) a->stack_c[o] = written[s] ? sc[(size_t)s * H + j] : 0.0;
            }

    /* ---------------- backward ---------------- */
    if (a->dh0 || a->dc0 || a->dx || a->dW || a->dbias) {
        if (a->d_top_h)
            for (int j = 0; j < H; ++j) ds_h[(size_t)p[T] * H + j] += a->d_top_h[(size_t)b * H + j];
        for (int t = T - 1; t >= 0; --t) {
            if (a->dy) {
                const double *dyt = a->dy + ((size_t)t * B + b) * H;
                for (int j = 0; j < H; ++j) ds_h[(size_t)p[t + 1] * H + j] += dyt[j];
            }
            double *dxt = a->dx ? a->dx + ((size_t)t * B + b) * I : NULL;
            if (!did[t]) {
                if (dxt) for (int k = 0; k < I; ++k) dxt[k] = 0.0;
                continue;
            }
            const int rd = p[t], wr = p[t] + 1;
            const double *gt = t_gate + (size_t)t * G;
            double *dhw = ds_h + (size_t)wr * H, *dcw = ds_c + (size_t)wr * H;
            double *dhr = ds_h + (size_t)rd * H, *dcr = ds_c + (size_t)rd * H;
            /* take the written state's gradient, then clear that slot */
            for (int j = 0; j < H; ++j) {
                const double dh = dhw[j], dcn = dcw[j];
                dhw[j] = 0.0;
                dcw[j] = 0.0;
                const double ig = gt[j], fg = gt[H + j], gg = gt[2 * H + j], og = gt[3 * H + j];
                const double tc = tanh(t_cn[(size_t)t * H + j]);
                const double dc = dcn + dh * og * (1.0 - tc * tc);
                dz[j] = dc * gg * ig * (1.0 - ig);
                dz[H + j] = dc * t_cr[(size_t)t * H + j] * fg * (1.0 - fg);
                dz[2 * H + j] = dc * ig * (1.0 - gg * gg);
                dz[3 * H + j] = dh * tc * og * (1.0 - og);
                dcr[j] += dc * fg; /* gradient of the cell state read */
            }
            /* dx_t = W[0:I] dz, dh_read = W[I:] dz */
            const double *xt = a->x + ((size_t)t * B + b) * I;
            for (int k = 0; k < K; ++k) {
                const double *Wk = a->W + (size_t)k * G;
                double s = 0.0;
                for (int n = 0; n < G; ++n) s += Wk[n] * dz[n];
                if (k < I) { if (dxt) dxt[k] = s; }
                else dhr[k - I] += s;
            }
            /* dW += [x_t ; h_read]^T dz, dbias += dz */
            if (a->dW)
                for (int k = 0; k < K; ++k) {
                    const double ak = k < I ? xt[k] : t_hr[(size_t)t * H + (k - I)];
                    double *dWk = a->dW + (size_t)k * G;
                    for (int n = 0; n < G; ++n) dWk[n] += ak * dz[n];
                }
            if (a->dbias)
                for (int n = 0; n < G; ++n) a->dbias[n] += dz[n];
        }
        for (int j = 0; j < H; ++j) {
            if (a->dh0) a->dh0[(size_t)b * H + j] = ds_h[j];
            if (a->dc0) a->dc0[(size_t)b * H + j] = ds_c[j];
        }
    }

done:
    free(sh); free(sc); free(tag); free(written); free(p);
    free(t_hr); free(t_cr); free(t_gate); free(t_cn); free(did);
    free(z); free(ds_h); free(ds_c); free(dz);
    return rc;
}

/*
 * Batched driver: runs every instance b in [0, B) independently (instances never
 * interact, Sec. 3). Arrays are C-ordered: x [T][B][I], ops [T][B], h0/c0 [B][H],
 * W [I+H][4H], bias [4H], d_top_h [B][H] (nullable), dy [T][B][H] (nullable).
 * Outputs (each nullable): p_traj [T+1][B], src [T+1][B], y [T][B][H],
 * stack_h/stack_c [T+1][B][H], dx [T][B][I], dh0/dc0 [B][H], dW [I+H][4H], dbias [4H].
 * dW and dbias are overwritten with the sum over instances: each thread sums a
 * contiguous block of instances in instance order, then the blocks are summed in order.
 * nthreads <= 0 uses one thread. Returns 0, or the first error code by instance order.
 */
int oracle_stacklstm(int T, int B, int I, int H, int mode,
                     const double *x, const int8_t *ops, const double *h0, const double *c0,
                     const double *W, const double *bias, const double *d_top_h, const double *dy,
                     int32_t *p_traj, int32_t *src, double *y, double *stack_h, double *stack_c,
                     double *dx, double *dh0, double *dc0, double *dW, double *dbias, int nthreads)
{
    if (T < 0 || B < 0 || I < 1 || H < 1 || (mode != ORACLE_HOMOGENIZED && mode != ORACLE_DEFINITION))
        return ORACLE_BAD_ARG;
    const size_t KG = (size_t)(I + H) * 4 * H, G = (size_t)4 * H;
    if (nthreads < 1) nthreads = 1;
    if (nthreads > B) nthreads = B > 0 ? B : 1;
    int *rcs = calloc((size_t)(B > 0 ? B : 1), sizeof(int));
    double *pdW = dW ? calloc((size_t)nthreads * KG, sizeof(double)) : NULL;
    double *pdb = dbias ? calloc((size_t)nthreads * G, sizeof(double)) : NULL;
    if (!rcs || (dW && !pdW) || (dbias && !pdb)) {
        free(rcs); free(pdW); free(pdb);
        return ORACLE_NOMEM;
    }
#ifdef _OPENMP
#pragma omp parallel for schedule(static, 1) num_threads(nthreads)
#endif
    for (int k = 0; k < nthreads; ++k) {
        const int b_lo = (int)((long long)B * k / nthreads), b_hi = (int)((long long)B * (k + 1) / nthreads);
        for (int b = b_lo; b < b_hi; ++b) {
            inst_args a = {T, B, I, H, mode, b, x, h0, c0, W, bias, d_top_h, dy, ops,
                           p_traj, src, y, stack_h, stack_c, dx, dh0, dc0,
                           pdW ? pdW + (size_t)k * KG : NULL, pdb ? pdb + (size_t)k * G : NULL};
            rcs[b] = run_instance(&a);
        }
    }
    int rc = ORACLE_OK;
    for (int b = 0; b < B && rc == ORACLE_OK; ++b) rc = rcs[b];
    if (dW) {
        memset(dW, 0, KG * sizeof(double));
        for (int k = 0; k < nthreads; ++k)
            for (size_t e = 0; e < KG; ++e) dW[e] += pdW[(size_t)k * KG + e];
    }
    if (dbias) {
        memset(dbias, 0, G * sizeof(double));
        for (int k = 0; k < nthreads; ++k)
            for (size_t e = 0; e < G; ++e) dbias[e] += pdb[(size_t)k * G + e];
    }
    free(rcs); free(pdW); free(pdb);
    return rc;
}

/*
 * Pointer trajectory and read provenance only (no cell arithmetic): the same explicit
 * stack of slot tags as above, for every instance. Fast enough for full-size batches.
 * Returns 0, or the first error code by instance order.
 */
int oracle_pointers(int T, int B, const int8_t *ops, int32_t *p_traj, int32_t *src)
{
    if (T < 0 || B < 0) return ORACLE_BAD_ARG;
    int32_t *tag = malloc((size_t)(T + 1) * sizeof(int32_t));
    if (!tag) return ORACLE_NOMEM;
    int rc = ORACLE_OK;
    for (int b = 0; b < B && rc == ORACLE_OK; ++b) {
        int p = 0;
        tag[0] = 0;
        for (int t = 0; t < T; ++t) {
            const int op = ops[(size_t)t * B + b];
            if (op != 1 && op != 0 && op != -1) { rc = ORACLE_BAD_OP; break; }
            if (p + op < 0) { rc = ORACLE_UNDERFLOW; break; }
            p_traj[(size_t)t * B + b] = p;
            src[(size_t)t * B + b] = tag[p];
            tag[p + 1] = t + 1; /* Algorithm 1: every step writes slot p + 1 */
            p += op;
        }
        p_traj[(size_t)T * B + b] = p;
        src[(size_t)T * B + b] = tag[p];
    }
    free(tag);
    return rc;
}
