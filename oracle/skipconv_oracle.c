/*
 * Skip-Convolution oracle: a plain, slow, double-precision CPU restatement of
 * the per-frame Skip-Conv layer step of Habibian et al., "Skip-Convolutions
 * for Efficient Video Processing" (CVPR 2021, arXiv 2104.11487).
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference leg of bench.py may load this library.  It shares
 * no code, header, table or helper with the CUDA library and never calls it.
 *
 * Conventions (all arrays are dense, row-major, caller-owned):
 *   x, x_prev, r : [n][h][w][c_in]          input frames (NHWC), double
 *   z            : [n][ho][wo][c_out]        output state (NHWC), double
 *   w            : [c_out][c_in/groups][k_h][k_w]   (the paper's c_o x c_i x k_h x k_w)
 *   score        : [n][ho][wo]               gate score per output location
 *   mask         : [n][nby][nbx]             block gate, 1 = process
 * with ho = (h + 2 pad - k_h)/stride + 1, nby = ceil(ho / block).
 *
 * Every loop below is the definition written out; nothing is blocked, fused
 * or reordered.  OpenMP (when compiled in) only splits outer independent
 * loops across threads.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef struct {
    int n;          /* independent streams processed side by side          */
    int c_in;
    int c_out;
    int h, w;       /* input frame height and width                         */
    int k_h, k_w;
    int stride;
    int pad;
    int groups;
    int block;      /* b: edge of the b x b gate blocks (Sec. 3.2, structured sparsity) */
    int gate;       /* 0 input-norm, mean over the support; 1 input-norm, sum;
                       2 output-norm (Eq. 7); 3 Gumbel gate (Eq. 8, inference) */
    double eps;
} oc_params;

enum { OC_GATE_INPUT_MEAN = 0, OC_GATE_INPUT_SUM = 1, OC_GATE_OUTPUT = 2, OC_GATE_GUMBEL = 3 };
enum { OC_ACT_NONE = 0, OC_ACT_RELU = 1, OC_ACT_SILU = 2 };

int oc_out_h(const oc_params* p) { return (p->h + 2 * p->pad - p->k_h) / p->stride + 1; }
int oc_out_w(const oc_params* p) { return (p->w + 2 * p->pad - p->k_w) / p->stride + 1; }
int oc_blocks_y(const oc_params* p) { return (oc_out_h(p) + p->block - 1) / p->block; }
int oc_blocks_x(const oc_params* p) { return (oc_out_w(p) + p->block - 1) / p->block; }

int oc_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void oc_set_num_threads(int t)
{
#ifdef _OPENMP
    if (t > 0) omp_set_num_threads(t);
#else
    (void)t;
#endif
}

/* index helpers */
static inline size_t ix_x(const oc_params* p, int n, int y, int x, int c)
{
    return (((size_t)n * p->h + y) * p->w + x) * p->c_in + c;
}
static inline size_t ix_z(const oc_params* p, int n, int i, int j, int o)
{
    return (((size_t)n * oc_out_h(p) + i) * oc_out_w(p) + j) * p->c_out + o;
}
static inline size_t ix_w(const oc_params* p, int o, int ci, int kh, int kw)
{
    int cpg = p->c_in / p->groups;
    return (((size_t)o * cpg + ci) * p->k_h + kh) * p->k_w + kw;
}

/* Input value at (n, y, x, c); positions outside the frame are the zero
 * padding of the convolution. */
static inline double at_or_zero(const oc_params* p, const double* a, int n, int y, int x, int c)
{
    if (y < 0 || y >= p->h || x < 0 || x >= p->w) return 0.0;
    return a[ix_x(p, n, y, x, c)];
}

/* ||w||_1 over all four dimensions of the layer's kernel (Eq. 7). */
double oc_weight_l1(const oc_params* p, const double* w)
{
    size_t nw = (size_t)p->c_out * (p->c_in / p->groups) * p->k_h * p->k_w;
    double s = 0.0;
    for (size_t i = 0; i < nw; ++i) s += fabs(w[i]);
    return s;
}

/* Residual frame r_t = x_t - x_{t-1} (Eq. 2). */
void oc_residual(const oc_params* p, const double* x_t, const double* x_prev, double* r)
{
    size_t nx = (size_t)p->n * p->h * p->w * p->c_in;
    for (size_t i = 0; i < nx; ++i) r[i] = x_t[i] - x_prev[i];
}

/* Norm-gate score at every output location.
 * Input-Norm gate (Eq. 5): the l1 norm of r_t over the kernel support of the
 * output location, i.e. |r| summed over all input channels and the k_h x k_w
 * window (p = 1), zero padding outside the frame.  Mode MEAN divides that sum
 * by the support size c_in*k_h*k_w; mode SUM keeps it.  Output-Norm gate
 * (Eq. 7): ||w||_1 times the same local sum. */
void oc_gate_scores(const oc_params* p, const double* r, double w_l1, double* score)
{
    const int ho = oc_out_h(p), wo = oc_out_w(p);
    const double support = (double)p->c_in * p->k_h * p->k_w;
#ifdef _OPENMP
#pragma omp parallel for collapse(2) schedule(static)
#endif
    for (int n = 0; n < p->n; ++n)
        for (int i = 0; i < ho; ++i)
            for (int j = 0; j < wo; ++j) {
                double s = 0.0;
                for (int kh = 0; kh < p->k_h; ++kh)
                    for (int kw = 0; kw < p->k_w; ++kw) {
                        int y = p->stride * i + kh - p->pad;
                        int x = p->stride * j + kw - p->pad;
                        for (int c = 0; c < p->c_in; ++c) s += fabs(at_or_zero(p, r, n, y, x, c));
                    }
                double v;
                if (p->gate == OC_GATE_INPUT_MEAN) v = s / support;
                else if (p->gate == OC_GATE_INPUT_SUM) v = s;
                else v = w_l1 * s;
                score[((size_t)n * ho + i) * wo + j] = v;
            }
}

/* Gumbel-gate score at every output location (Eq. 8 at inference): the gate
 * function f(r; phi) is a convolution of r with a single output channel and
 * the layer's kernel size, stride and zero padding, plus its bias:
 *   f(i,j) = phi_bias + sum_{c,kh,kw} phi[c][kh][kw] r[c, s i + kh - pad, s j + kw - pad].
 * The gate round(sigmoid(f)) is 1 exactly when f > 0, i.e. the block gate
 * below with eps = 0.  phi is [c_in][k_h][k_w]. */
void oc_gumbel_scores(const oc_params* p, const double* r, const double* phi, double phi_bias, double* score)
{
    const int ho = oc_out_h(p), wo = oc_out_w(p);
#ifdef _OPENMP
#pragma omp parallel for collapse(2) schedule(static)
#endif
    for (int n = 0; n < p->n; ++n)
        for (int i = 0; i < ho; ++i)
            for (int j = 0; j < wo; ++j) {
                double f = phi_bias;
                for (int c = 0; c < p->c_in; ++c)
                    for (int kh = 0; kh < p->k_h; ++kh)
                        for (int kw = 0; kw < p->k_w; ++kw) {
                            int y = p->stride * i + kh - p->pad;
                            int x = p->stride * j + kw - p->pad;
                            f += phi[((size_t)c * p->k_h + kh) * p->k_w + kw] * at_or_zero(p, r, n, y, x, c);
                        }
                score[((size_t)n * ho + i) * wo + j] = f;
            }
}

/* The gate score of the layer's gate mode. */
static void gate_scores_of(const oc_params* p, const double* w, const double* r, const double* phi, double phi_bias,
                           double* score)
{
    if (p->gate == OC_GATE_GUMBEL) oc_gumbel_scores(p, r, phi, phi_bias, score);
    else oc_gate_scores(p, r, p->gate == OC_GATE_OUTPUT ? oc_weight_l1(p, w) : 0.0, score);
}

/* Block gate (Sec. 3.2, structured sparsity): the pixel gate is
 * round(sigmoid(score - eps)), which is 1 exactly when score > eps; max-pooling
 * it with kernel and stride b opens a block when any of its locations is open.
 * Edge blocks cover the remaining locations (ceil mode).  force = 1 opens every
 * block (first frame after a reset, Sec. 3.1; or the all-ones dense mode). */
void oc_block_gate(const oc_params* p, const double* score, int force, unsigned char* mask)
{
    const int ho = oc_out_h(p), wo = oc_out_w(p);
    const int nby = oc_blocks_y(p), nbx = oc_blocks_x(p), b = p->block;
    for (int n = 0; n < p->n; ++n)
        for (int by = 0; by < nby; ++by)
            for (int bx = 0; bx < nbx; ++bx) {
                int open = 0;
                for (int i = by * b; i < by * b + b && i < ho; ++i)
                    for (int j = bx * b; j < bx * b + b && j < wo; ++j)
                        if (score[((size_t)n * ho + i) * wo + j] > p->eps) open = 1;
                mask[((size_t)n * nby + by) * nbx + bx] = (unsigned char)(force ? 1 : open);
            }
}

/* (w * r) at one output location and output channel (Eq. 1 applied to r). */
static double conv_at(const oc_params* p, const double* w, const double* r, int n, int i, int j, int o)
{
    const int cpg = p->c_in / p->groups;
    const int opg = p->c_out / p->groups;
    const int g = o / opg;
    double acc = 0.0;
    for (int ci = 0; ci < cpg; ++ci)
        for (int kh = 0; kh < p->k_h; ++kh)
            for (int kw = 0; kw < p->k_w; ++kw) {
                int y = p->stride * i + kh - p->pad;
                int x = p->stride * j + kw - p->pad;
                acc += w[ix_w(p, o, ci, kh, kw)] * at_or_zero(p, r, n, y, x, g * cpg + ci);
            }
    return acc;
}

/* Standard convolution z = w * x + bias (Eq. 1), every location. */
void oc_dense_conv(const oc_params* p, const double* w, const double* bias, const double* x, double* z)
{
    const int ho = oc_out_h(p), wo = oc_out_w(p);
#ifdef _OPENMP
#pragma omp parallel for collapse(2) schedule(static)
#endif
    for (int n = 0; n < p->n; ++n)
        for (int i = 0; i < ho; ++i)
            for (int j = 0; j < wo; ++j)
                for (int o = 0; o < p->c_out; ++o)
                    z[ix_z(p, n, i, j, o)] = (bias ? bias[o] : 0.0) + conv_at(p, w, x, n, i, j, o);
}

/* State after a reset: x_{t-1} = 0 and z = bias, so the next residual is the
 * frame itself and the next step is a key frame (Sec. 3.1). */
void oc_reset(const oc_params* p, const double* bias, double* x_prev, double* z)
{
    size_t nx = (size_t)p->n * p->h * p->w * p->c_in;
    size_t nz = (size_t)p->n * oc_out_h(p) * oc_out_w(p) * p->c_out;
    memset(x_prev, 0, nx * sizeof(double));
    for (size_t i = 0; i < nz; ++i) z[i] = bias ? bias[i % p->c_out] : 0.0;
}

/* One Skip-Conv step (Eq. 3):  z~_t = z~_{t-1} + g(r_t) (.) (w * r_t),
 * r_t = x_t - x_{t-1}; ungated locations keep z~_{t-1}; then x_{t-1} <- x_t.
 * phi / phi_bias: the Gumbel gate's function (gate mode 3), else unused.
 * force = 1 opens every gate (key frame or dense mode).
 * score_out ([n][ho][wo]) and mask_out ([n][nby][nbx]) may be NULL.
 * Returns the number of open blocks, or -1 on allocation failure. */
long oc_step(const oc_params* p, const double* w, const double* phi, double phi_bias, const double* x_t,
             double* x_prev, double* z, int force, double* score_out, unsigned char* mask_out)
{
    const int ho = oc_out_h(p), wo = oc_out_w(p);
    const int nby = oc_blocks_y(p), nbx = oc_blocks_x(p), b = p->block;
    size_t nx = (size_t)p->n * p->h * p->w * p->c_in;
    double* r = (double*)malloc(nx * sizeof(double));
    double* score = score_out ? score_out : (double*)malloc((size_t)p->n * ho * wo * sizeof(double));
    unsigned char* mask = mask_out ? mask_out : (unsigned char*)malloc((size_t)p->n * nby * nbx);
    if (!r || !score || !mask) {
        free(r);
        if (!score_out) free(score);
        if (!mask_out) free(mask);
        return -1;
    }
    oc_residual(p, x_t, x_prev, r);
    gate_scores_of(p, w, r, phi, phi_bias, score);
    oc_block_gate(p, score, force, mask);
#ifdef _OPENMP
#pragma omp parallel for collapse(2) schedule(dynamic)
#endif
    for (int n = 0; n < p->n; ++n)
        for (int i = 0; i < ho; ++i)
            for (int j = 0; j < wo; ++j) {
                if (!mask[((size_t)n * nby + i / b) * nbx + j / b]) continue;
                for (int o = 0; o < p->c_out; ++o) z[ix_z(p, n, i, j, o)] += conv_at(p, w, r, n, i, j, o);
            }
    memcpy(x_prev, x_t, nx * sizeof(double));
    long open = 0;
    for (size_t k = 0; k < (size_t)p->n * nby * nbx; ++k) open += mask[k];
    free(r);
    if (!score_out) free(score);
    if (!mask_out) free(mask);
    return open;
}

/* Warp T of Sec. 3.4 (Eq. 10-11): out(n, y, x, c) = in sampled at
 * (y + dy, x + dx), (dy, dx) = flow[n][y][x], by bilinear interpolation of the
 * four surrounding pixels; a pixel outside the frame contributes zero.  in and
 * out are [n][H][W][C]; flow is [n][H][W][2] (dy, dx) in pixels. */
void oc_warp(int n, int H, int W, int C, const double* flow, const double* in, double* out)
{
#ifdef _OPENMP
#pragma omp parallel for collapse(2) schedule(static)
#endif
    for (int ni = 0; ni < n; ++ni)
        for (int y = 0; y < H; ++y)
            for (int x = 0; x < W; ++x) {
                const double* f = flow + (((size_t)ni * H + y) * W + x) * 2;
                const double sy = y + f[0], sx = x + f[1];
                const double fy = floor(sy), fx = floor(sx);
                const double ay = sy - fy, ax = sx - fx;
                const int y0 = (int)fy, x0 = (int)fx;
                const int ys[4] = {y0, y0, y0 + 1, y0 + 1}, xs[4] = {x0, x0 + 1, x0, x0 + 1};
                const double wt[4] = {(1.0 - ay) * (1.0 - ax), (1.0 - ay) * ax, ay * (1.0 - ax), ay * ax};
                for (int c = 0; c < C; ++c) {
                    double v = 0.0;
                    for (int q = 0; q < 4; ++q)
                        if (ys[q] >= 0 && ys[q] < H && xs[q] >= 0 && xs[q] < W)
                            v += wt[q] * in[(((size_t)ni * H + ys[q]) * W + xs[q]) * C + c];
                    out[(((size_t)ni * H + y) * W + x) * C + c] = v;
                }
            }
}

/* Skip-Conv step with a warped residual (Sec. 3.4, Eq. 10-11): the residual
 * is taken against the previous input warped by T,
 *     r_t = x_t - T(x_{t-1}),
 * and the output is decoded by warping the previous output with the same
 * flow before adding the gated convolution of the residual,
 *     z~_t = T~(z~_{t-1}) + g(r_t) (.) (w * r_t),
 * then x_{t-1} <- x_t.  T~ applies the flow on the output grid, so the layer
 * must keep the frame size (stride 1, ho = h, wo = w).  The gate, blocks and
 * force are those of oc_step.  Returns the number of open blocks, -1 on
 * allocation failure, -2 when the output grid differs from the input grid. */
long oc_step_warped(const oc_params* p, const double* w, const double* phi, double phi_bias, const double* x_t,
                    double* x_prev, double* z, const double* flow, int force, double* score_out,
                    unsigned char* mask_out)
{
    const int ho = oc_out_h(p), wo = oc_out_w(p);
    if (p->stride != 1 || ho != p->h || wo != p->w) return -2;
    const int nby = oc_blocks_y(p), nbx = oc_blocks_x(p), b = p->block;
    size_t nx = (size_t)p->n * p->h * p->w * p->c_in;
    size_t nz = (size_t)p->n * ho * wo * p->c_out;
    double* tx = (double*)malloc(nx * sizeof(double));
    double* r = (double*)malloc(nx * sizeof(double));
    double* zw = (double*)malloc(nz * sizeof(double));
    double* score = score_out ? score_out : (double*)malloc((size_t)p->n * ho * wo * sizeof(double));
    unsigned char* mask = mask_out ? mask_out : (unsigned char*)malloc((size_t)p->n * nby * nbx);
    if (!tx || !r || !zw || !score || !mask) {
        free(tx);
        free(r);
        free(zw);
        if (!score_out) free(score);
        if (!mask_out) free(mask);
        return -1;
    }
    oc_warp(p->n, p->h, p->w, p->c_in, flow, x_prev, tx);    /* T(x_{t-1}) */
    oc_residual(p, x_t, tx, r);                              /* r_t = x_t - T(x_{t-1}) */
    gate_scores_of(p, w, r, phi, phi_bias, score);
    oc_block_gate(p, score, force, mask);
    oc_warp(p->n, ho, wo, p->c_out, flow, z, zw);            /* T~(z~_{t-1}) */
    memcpy(z, zw, nz * sizeof(double));
#ifdef _OPENMP
#pragma omp parallel for collapse(2) schedule(dynamic)
#endif
    for (int n = 0; n < p->n; ++n)
        for (int i = 0; i < ho; ++i)
            for (int j = 0; j < wo; ++j) {
                if (!mask[((size_t)n * nby + i / b) * nbx + j / b]) continue;
                for (int o = 0; o < p->c_out; ++o) z[ix_z(p, n, i, j, o)] += conv_at(p, w, r, n, i, j, o);
            }
    memcpy(x_prev, x_t, nx * sizeof(double));
    long open = 0;
    for (size_t k = 0; k < (size_t)p->n * nby * nbx; ++k) open += mask[k];
    free(tx);
    free(r);
    free(zw);
    if (!score_out) free(score);
    if (!mask_out) free(mask);
    return open;
}

/* The same step, with z kept only at n_samples chosen output locations
 * (z_samples is [n_samples][c_out], locations given as (n, i, j) triples).
 * The gate is evaluated over the whole frame exactly as in oc_step, so the
 * sampled z follows the same recurrence as the full one. */
long oc_step_sampled(const oc_params* p, const double* w, const double* phi, double phi_bias, const double* x_t,
                     double* x_prev, int n_samples, const int* sample_nij, double* z_samples, int force,
                     unsigned char* mask_out)
{
    const int ho = oc_out_h(p), wo = oc_out_w(p);
    const int nby = oc_blocks_y(p), nbx = oc_blocks_x(p), b = p->block;
    size_t nx = (size_t)p->n * p->h * p->w * p->c_in;
    double* r = (double*)malloc(nx * sizeof(double));
    double* score = (double*)malloc((size_t)p->n * ho * wo * sizeof(double));
    unsigned char* mask = mask_out ? mask_out : (unsigned char*)malloc((size_t)p->n * nby * nbx);
    if (!r || !score || !mask) {
        free(r);
        free(score);
        if (!mask_out) free(mask);
        return -1;
    }
    oc_residual(p, x_t, x_prev, r);
    gate_scores_of(p, w, r, phi, phi_bias, score);
    oc_block_gate(p, score, force, mask);
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic)
#endif
    for (int s = 0; s < n_samples; ++s) {
        int n = sample_nij[3 * s], i = sample_nij[3 * s + 1], j = sample_nij[3 * s + 2];
        if (!mask[((size_t)n * nby + i / b) * nbx + j / b]) continue;
        for (int o = 0; o < p->c_out; ++o) z_samples[(size_t)s * p->c_out + o] += conv_at(p, w, r, n, i, j, o);
    }
    memcpy(x_prev, x_t, nx * sizeof(double));
    long open = 0;
    for (size_t k = 0; k < (size_t)p->n * nby * nbx; ++k) open += mask[k];
    free(r);
    free(score);
    if (!mask_out) free(mask);
    return open;
}

/* Round a double to the nearest bfloat16 value (ties to even), returned as a
 * double.  bfloat16 keeps 8 significant bits and the float32 exponent range;
 * values beyond its largest finite value become infinities.  Used where a
 * stack hands a layer's output to the next layer at bfloat16 precision. */
double oc_round_bf16(double v)
{
    if (v == 0.0 || isnan(v) || isinf(v)) return v;
    int e;
    (void)frexp(fabs(v), &e);                 /* |v| = m * 2^e, m in [0.5, 1) */
    /* float32 normal range: exponent e-1 >= -126, i.e. e >= -125; below it
     * the spacing stays at 2^-133 (bfloat16 subnormals). */
    int eff = e < -125 ? -125 : e;
    double ulp = ldexp(1.0, eff - 8);          /* 8 significant bits */
    double q = fabs(v) / ulp;
    double fl = floor(q);
    double rem = q - fl;
    double res;
    if (rem > 0.5) res = fl + 1.0;
    else if (rem < 0.5) res = fl;
    else res = (fmod(fl, 2.0) == 0.0) ? fl : fl + 1.0;
    res *= ulp;
    if (res > 3.3895313892515355e38) res = INFINITY;  /* largest finite bfloat16 */
    return v < 0 ? -res : res;
}

/* Round a double to the nearest float32 value (ties to even), as a double. */
double oc_round_f32(double v) { return (double)(float)v; }

/* Layer output handed to the next layer: y = act(z [+ shortcut]), computed in
 * double, then rounded to the layer's storage precision (0: none, 1: float32,
 * 2: bfloat16).  z is pre-activation (Sec. 3.1). */
void oc_layer_output(size_t count, const double* z, const double* shortcut, int act, int round_mode, double* y)
{
    for (size_t k = 0; k < count; ++k) {
        double v = z[k] + (shortcut ? shortcut[k] : 0.0);
        if (act == OC_ACT_RELU) v = v > 0.0 ? v : 0.0;
        else if (act == OC_ACT_SILU) v = v / (1.0 + exp(-v));
        if (round_mode == 1) v = oc_round_f32(v);
        else if (round_mode == 2) v = oc_round_bf16(v);
        y[k] = v;
    }
}
