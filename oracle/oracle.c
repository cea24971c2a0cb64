/*
 * Plain, slow CPU oracle for 1xN pruning and the 1xN-pruned convolution.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is compiled into liboracle.so and is
 * loaded by tests/, by __graft_entry__.smoke() and by the cpu_baseline /
 * reference leg of bench.py.  The product library never links, loads or calls
 * it, and it shares no code, header, table or helper with the CUDA path.
 *
 * Everything is written the way the paper states it, in double precision,
 * with no blocking, fusion or reordering beyond what the definitions say:
 *
 *   Notation (Sec. 3.1): layer weight W in R^{n x m x h x w}; n = output
 *   channels (C_out), m = input channels (C_in), h x w = kernel (KH x KW).
 *   Sec. 3.2 reshapes W as Omega in R^{m x n}, Omega[k, j] = W[j, k, :, :],
 *   and partitions each row of Omega into n/N col-groups of N consecutive
 *   output kernels: block (k, g) = Omega[k, gN : (g+1)N]  (0-based).
 *
 *   Two block granularities are provided (reading C1):
 *     ORACLE_GRAN_TAP    : one block per (g, c, kh, kw), N weights; the block
 *                          index is k = (kh*KW + kw)*C_in + c (tap-major).
 *     ORACLE_GRAN_KERNEL : the paper's block of Sec. 3.2, one per (g, c),
 *                          N*KH*KW weights.  A kept (g, c) keeps all KH*KW
 *                          tap indices of channel c.
 *   In both, the stored mask is expanded to the tap index space: mask[g][k]
 *   for k in [0, KH*KW*C_in) (the transpose of the paper's T in R^{m x n/N}).
 *
 *   The importance of a block is its l1 norm (Eq. 1, Eq. 4); the blocks with
 *   the largest norms, top (1-p) of them, are kept (the closed-form solution
 *   stated after Eq. 5).  The kept count is round-half-up((1-p) * #blocks)
 *   in exact integer arithmetic (reading C3); ties in the norm go to the
 *   lower block index (reading C4).
 *
 *   Filter rearrangement (Sec. 3.3): filters are re-ordered by their l1 norm
 *   in decreasing order (stable), and the next layer's input channels are
 *   permuted the same way.
 *
 *   BSR encoding (Sec. 3.4): D in R^{t x N} stacks the kept blocks col-group
 *   by col-group, I in Z^t holds each block's row (index) k, and
 *   P in Z^{n/N+1} holds each col-group's start offset; 0-based, so
 *   P[G] = t (reading C2).
 *
 *   Output (Eq. 6, and its block-wise form Eq. 7, read as
 *   Y[:, gN:(g+1)N] = sum_{z=P[g]}^{P[g+1]-1} X[:, I[z]] * D[z, :]):
 *   a direct NHWC convolution with zero padding, stride and dilation, with an
 *   optional per-output-channel bias and ReLU.
 *
 *   Fine-tuning of the pruned network (Sec. 4.1) with the mask held fixed:
 *   the gradients of that output with respect to the input and to the kept
 *   weights, written from the definition of the convolution.
 *
 * Build: gcc -O2 -fopenmp -ffp-contract=off -shared -fPIC oracle.c
 * (the only parallelism is an OpenMP loop over independent output pixels).
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <math.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORACLE_GRAN_TAP 0
#define ORACLE_GRAN_KERNEL 1

/* ------------------------------------------------------------------ */
/* Keep count (Eq. 1 constraint ||T||_0 / K = 1 - p; reading C3).       */
/* ------------------------------------------------------------------ */
int64_t oracle_keep_count(int64_t total_blocks, double rate)
{
    /* rate is taken at a resolution of 1e-6, then
     * keep = floor(total * (1e6 - r6) / 1e6 + 1/2), all in int64. */
    int64_t r6 = llround(rate * 1000000.0);
    if (r6 < 0) r6 = 0;
    if (r6 > 1000000) r6 = 1000000;
    return (total_blocks * (1000000 - r6) + 500000) / 1000000;
}

/* W is OIHW fp32: W[o][c][kh][kw]. */
static double w_at(const float *W, int C_in, int KH, int KW,
                   int o, int c, int kh, int kw)
{
    return (double)W[(((int64_t)o * C_in + c) * KH + kh) * KW + kw];
}

/* ------------------------------------------------------------------ */
/* Block l1 norms (Eq. 4 / Eq. 5 with L = l1 norm).                     */
/* score layout: [G][nb], nb = KH*KW*C_in (TAP) or C_in (KERNEL).       */
/* Summation order: n ascending; in KERNEL mode n, then kh, then kw.    */
/* ------------------------------------------------------------------ */
void oracle_block_scores(const float *W, int C_out, int C_in, int KH, int KW,
                         int N, int gran, double *score)
{
    int G = C_out / N;
    if (gran == ORACLE_GRAN_TAP) {
        int K = KH * KW * C_in;
        for (int g = 0; g < G; g++)
            for (int k = 0; k < K; k++) {
                int tap = k / C_in, c = k % C_in;
                int kh = tap / KW, kw = tap % KW;
                double s = 0.0;
                for (int n = 0; n < N; n++)
                    s += fabs(w_at(W, C_in, KH, KW, g * N + n, c, kh, kw));
                score[(int64_t)g * K + k] = s;
            }
    } else {
        for (int g = 0; g < G; g++)
            for (int c = 0; c < C_in; c++) {
                double s = 0.0;
                for (int n = 0; n < N; n++)
                    for (int kh = 0; kh < KH; kh++)
                        for (int kw = 0; kw < KW; kw++)
                            s += fabs(w_at(W, C_in, KH, KW, g * N + n, c, kh, kw));
                score[(int64_t)g * C_in + c] = s;
            }
    }
}

/* Ordering of blocks for the top-(1-p) selection: larger norm first, then
 * the lower block index (g * nb + b). */
typedef struct { double s; int64_t idx; } ranked;

static int ranked_cmp(const void *a, const void *b)
{
    const ranked *x = (const ranked *)a, *y = (const ranked *)b;
    if (x->s > y->s) return -1;
    if (x->s < y->s) return 1;
    return (x->idx < y->idx) ? -1 : (x->idx > y->idx);
}

/* ------------------------------------------------------------------ */
/* 1xN pruning mask (Eq. 4 / Eq. 5 and the solution after Eq. 5).       */
/* mask: [G][KH*KW*C_in] in the tap index space.  Returns 0 on success. */
/* ------------------------------------------------------------------ */
int oracle_prune(const float *W, int C_out, int C_in, int KH, int KW, int N,
                 double rate, int gran, uint8_t *mask, int64_t *kept)
{
    if (N < 1 || C_out % N != 0 || rate < 0.0 || rate > 1.0) return 1;
    int G = C_out / N;
    int K = KH * KW * C_in;
    int nb = (gran == ORACLE_GRAN_TAP) ? K : C_in;
    int64_t total = (int64_t)G * nb;
    double *score = (double *)malloc(sizeof(double) * total);
    ranked *r = (ranked *)malloc(sizeof(ranked) * total);
    oracle_block_scores(W, C_out, C_in, KH, KW, N, gran, score);
    for (int64_t i = 0; i < total; i++) { r[i].s = score[i]; r[i].idx = i; }
    qsort(r, total, sizeof(ranked), ranked_cmp);
    int64_t keep = oracle_keep_count(total, rate);

    memset(mask, 0, (size_t)G * K);
    for (int64_t i = 0; i < keep; i++) {
        int64_t g = r[i].idx / nb, b = r[i].idx % nb;
        if (gran == ORACLE_GRAN_TAP) {
            mask[g * K + b] = 1;
        } else {
            for (int tap = 0; tap < KH * KW; tap++)
                mask[g * K + (int64_t)tap * C_in + b] = 1;
        }
    }
    *kept = keep;
    free(score);
    free(r);
    return 0;
}

/* ------------------------------------------------------------------ */
/* Filter rearrangement (Sec. 3.3).                                     */
/* W_l: [C_out][C_in][KH][KW], permuted in place along C_out.           */
/* W_next (nullable): [C_out_next][C_out][KH_n][KW_n], permuted in place */
/* along its input-channel dim.  perm[o'] = original index of the filter */
/* that lands at position o'.                                            */
/* ------------------------------------------------------------------ */
int oracle_rearrange(float *W_l, int C_out, int C_in, int KH, int KW,
                     float *W_next, int C_out_next, int KH_n, int KW_n,
                     int32_t *perm)
{
    int64_t fs = (int64_t)C_in * KH * KW;
    ranked *r = (ranked *)malloc(sizeof(ranked) * C_out);
    for (int o = 0; o < C_out; o++) {
        double s = 0.0;                    /* l1 of filter o, (c, kh, kw) row-major */
        for (int64_t e = 0; e < fs; e++) s += fabs((double)W_l[o * fs + e]);
        r[o].s = s;
        r[o].idx = o;
    }
    qsort(r, C_out, sizeof(ranked), ranked_cmp);   /* decreasing, stable by index */
    for (int o = 0; o < C_out; o++) perm[o] = (int32_t)r[o].idx;

    float *tmp = (float *)malloc(sizeof(float) * fs * C_out);
    memcpy(tmp, W_l, sizeof(float) * fs * C_out);
    for (int o = 0; o < C_out; o++)
        memcpy(W_l + o * fs, tmp + (int64_t)perm[o] * fs, sizeof(float) * fs);
    free(tmp);

    if (W_next) {
        int64_t ks = (int64_t)KH_n * KW_n;
        int64_t ns = (int64_t)C_out * ks;       /* one next-layer filter */
        float *t2 = (float *)malloc(sizeof(float) * ns);
        for (int j = 0; j < C_out_next; j++) {
            memcpy(t2, W_next + j * ns, sizeof(float) * ns);
            for (int o = 0; o < C_out; o++)
                memcpy(W_next + j * ns + o * ks, t2 + (int64_t)perm[o] * ks,
                       sizeof(float) * ks);
        }
        free(t2);
    }
    free(r);
    return 0;
}

/* Round-to-nearest-even of an fp32 value to bfloat16 (returned as the
 * upper 16 bits).  Textbook bit method: add 0x7fff plus the lowest kept
 * bit, then drop the low 16 bits.  Inputs here are finite. */
static uint16_t f32_to_bf16_rne(float f)
{
    uint32_t u;
    memcpy(&u, &f, 4);
    uint32_t lsb = (u >> 16) & 1u;
    u += 0x7fffu + lsb;
    return (uint16_t)(u >> 16);
}

void oracle_round_bf16(const float *in, float *out, int64_t n)
{
    for (int64_t i = 0; i < n; i++) {
        uint32_t u = (uint32_t)f32_to_bf16_rne(in[i]) << 16;
        memcpy(&out[i], &u, 4);
    }
}

/* ------------------------------------------------------------------ */
/* BSR encoding (Sec. 3.4, Fig. 3).  dtype 0: D fp32; 1: D bf16 (RNE). */
/* P: [G+1]; I: [t]; D: [t][N].  Returns t, or -1 if t_cap is short.    */
/* ------------------------------------------------------------------ */
int64_t oracle_pack(const float *W, const uint8_t *mask, int C_out, int C_in,
                    int KH, int KW, int N, int dtype, int32_t *P, int32_t *I,
                    void *D, int64_t t_cap)
{
    int G = C_out / N;
    int K = KH * KW * C_in;
    int64_t z = 0;
    for (int g = 0; g < G; g++) {
        P[g] = (int32_t)z;                       /* start of col-group g */
        for (int k = 0; k < K; k++) {
            if (!mask[(int64_t)g * K + k]) continue;
            if (z >= t_cap) return -1;
            int tap = k / C_in, c = k % C_in, kh = tap / KW, kw = tap % KW;
            I[z] = k;                            /* row index of the block */
            for (int n = 0; n < N; n++) {
                float v = (float)w_at(W, C_in, KH, KW, g * N + n, c, kh, kw);
                if (dtype == 0) ((float *)D)[z * N + n] = v;
                else ((uint16_t *)D)[z * N + n] = f32_to_bf16_rne(v);
            }
            z++;
        }
    }
    P[G] = (int32_t)z;                           /* fictitious last entry */
    return z;
}

/* Inverse of the encoding: dense masked weights W (OIHW fp32) from fp32 D. */
void oracle_unpack(const int32_t *P, const int32_t *I, const float *D,
                   int C_out, int C_in, int KH, int KW, int N, float *W)
{
    int G = C_out / N;
    memset(W, 0, sizeof(float) * (size_t)C_out * C_in * KH * KW);
    for (int g = 0; g < G; g++)
        for (int32_t z = P[g]; z < P[g + 1]; z++) {
            int k = I[z], tap = k / C_in, c = k % C_in, kh = tap / KW, kw = tap % KW;
            for (int n = 0; n < N; n++)
                W[(((int64_t)(g * N + n) * C_in + c) * KH + kh) * KW + kw] = D[(int64_t)z * N + n];
        }
}

/* Output geometry of a padded, strided, dilated convolution. */
static int out_size(int in, int k, int s, int p, int d)
{
    return (in + 2 * p - d * (k - 1) - 1) / s + 1;
}

typedef struct {
    int B, H, W, C_in, C_out, KH, KW;
    int sh, sw, ph, pw, dh, dw;
    int relu;
} oracle_geom;

/* Activation after the bias: 0 none, 1 ReLU max(s, 0), 2 ReLU6            */
/* min(max(s, 0), 6) (MobileNet-V2's activation).                           */
static double act(double s, int kind)
{
    if (kind >= 1 && s < 0.0) s = 0.0;
    if (kind == 2 && s > 6.0) s = 6.0;
    return s;
}

/* x value at NHWC input position, zero outside the image (zero padding). */
static double x_at(const float *x, const oracle_geom *g, int b, int ih, int iw, int c)
{
    if (ih < 0 || ih >= g->H || iw < 0 || iw >= g->W) return 0.0;
    return (double)x[(((int64_t)b * g->H + ih) * g->W + iw) * g->C_in + c];
}

/* ------------------------------------------------------------------ */
/* Eq. 6: masked direct convolution, y[b,oh,ow,o] =                    */
/*   bias[o] + sum_{kh,kw,c} mask[o/N][(kh*KW+kw)*C_in+c] * W[o,c,kh,kw] */
/*                        * x[b, oh*sh - ph + kh*dh, ow*sw - pw + kw*dw, c] */
/* then the activation g->relu (1 ReLU, 2 ReLU6).                          */
/* absacc[...] = sum |mask*W*x| + |bias| (C12).                            */
/* pix (nullable): list of npix flattened output pixels b*Ho*Wo+oh*Wo+ow; */
/* y/absacc are then [npix][C_out], else [B][Ho][Wo][C_out].             */
/* mask may be NULL (dense).                                             */
/* ------------------------------------------------------------------ */
void oracle_conv_masked(const float *x, const float *W, const uint8_t *mask,
                        const float *bias, const oracle_geom *g, int N,
                        const int64_t *pix, int64_t npix,
                        double *y, double *absacc)
{
    int Ho = out_size(g->H, g->KH, g->sh, g->ph, g->dh);
    int Wo = out_size(g->W, g->KW, g->sw, g->pw, g->dw);
    int64_t total = pix ? npix : (int64_t)g->B * Ho * Wo;
    int K = g->KH * g->KW * g->C_in;
#pragma omp parallel for schedule(dynamic, 16)
    for (int64_t q = 0; q < total; q++) {
        int64_t p = pix ? pix[q] : q;
        int b = (int)(p / ((int64_t)Ho * Wo));
        int oh = (int)((p / Wo) % Ho), ow = (int)(p % Wo);
        for (int o = 0; o < g->C_out; o++) {
            double s = bias ? (double)bias[o] : 0.0;
            double a = bias ? fabs((double)bias[o]) : 0.0;
            for (int kh = 0; kh < g->KH; kh++)
                for (int kw = 0; kw < g->KW; kw++)
                    for (int c = 0; c < g->C_in; c++) {
                        int k = (kh * g->KW + kw) * g->C_in + c;
                        if (mask && !mask[(int64_t)(o / N) * K + k]) continue;
                        double w = w_at(W, g->C_in, g->KH, g->KW, o, c, kh, kw);
                        double v = x_at(x, g, b, oh * g->sh - g->ph + kh * g->dh,
                                        ow * g->sw - g->pw + kw * g->dw, c);
                        s += w * v;
                        a += fabs(w * v);
                    }
            s = act(s, g->relu);
            y[q * g->C_out + o] = s;
            if (absacc) absacc[q * g->C_out + o] = a;
        }
    }
}

/* ------------------------------------------------------------------ */
/* Eq. 7: the block-wise decode straight from (P, I, D).  For each      */
/* output pixel and col-group g, Y[pix, gN:(g+1)N] =                    */
/*   sum_{z=P[g]}^{P[g+1]-1} X[pix, I[z]] * D[z, :]  (+ bias, ReLU).     */
/* D is fp32 (dtype 0) or bf16 bits (dtype 1).  Same pix convention.     */
/* ------------------------------------------------------------------ */
void oracle_conv_bsr(const float *x, const int32_t *P, const int32_t *I,
                     const void *D, int dtype, const float *bias,
                     const oracle_geom *g, int N, const int64_t *pix,
                     int64_t npix, double *y)
{
    int Ho = out_size(g->H, g->KH, g->sh, g->ph, g->dh);
    int Wo = out_size(g->W, g->KW, g->sw, g->pw, g->dw);
    int64_t total = pix ? npix : (int64_t)g->B * Ho * Wo;
    int G = g->C_out / N;
#pragma omp parallel for schedule(dynamic, 16)
    for (int64_t q = 0; q < total; q++) {
        int64_t p = pix ? pix[q] : q;
        int b = (int)(p / ((int64_t)Ho * Wo));
        int oh = (int)((p / Wo) % Ho), ow = (int)(p % Wo);
        for (int gi = 0; gi < G; gi++) {
            for (int n = 0; n < N; n++) {
                double s = bias ? (double)bias[gi * N + n] : 0.0;
                for (int32_t z = P[gi]; z < P[gi + 1]; z++) {
                    int k = I[z];
                    int tap = k / g->C_in, c = k % g->C_in;
                    int kh = tap / g->KW, kw = tap % g->KW;
                    double v = x_at(x, g, b, oh * g->sh - g->ph + kh * g->dh,
                                    ow * g->sw - g->pw + kw * g->dw, c);
                    double d;
                    if (dtype == 0) {
                        d = (double)((const float *)D)[(int64_t)z * N + n];
                    } else {
                        uint32_t u = (uint32_t)((const uint16_t *)D)[(int64_t)z * N + n] << 16;
                        float f;
                        memcpy(&f, &u, 4);
                        d = (double)f;
                    }
                    s += v * d;
                }
                s = act(s, g->relu);
                y[q * g->C_out + gi * N + n] = s;
            }
        }
    }
}

/* ------------------------------------------------------------------ */
/* Depthwise convolution (dense; MobileNet-V2's 3x3 between the expand  */
/* and project 1x1 convolutions): channel c of the output reads only     */
/* channel c of the input,                                               */
/*   y[b,oh,ow,c] = act(bias[c] + sum_{kh,kw} W[c,kh,kw]                 */
/*                  * x[b, oh*sh - ph + kh*dh, ow*sw - pw + kw*dw, c]).   */
/* g->C_in == g->C_out == C; W is [C][KH][KW]; y is [B][Ho][Wo][C].      */
/* ------------------------------------------------------------------ */
void oracle_dwconv(const float *x, const float *W, const float *bias,
                   const oracle_geom *g, double *y)
{
    int Ho = out_size(g->H, g->KH, g->sh, g->ph, g->dh);
    int Wo = out_size(g->W, g->KW, g->sw, g->pw, g->dw);
    int64_t total = (int64_t)g->B * Ho * Wo;
#pragma omp parallel for schedule(dynamic, 16)
    for (int64_t p = 0; p < total; p++) {
        int b = (int)(p / ((int64_t)Ho * Wo));
        int oh = (int)((p / Wo) % Ho), ow = (int)(p % Wo);
        for (int c = 0; c < g->C_in; c++) {
            double s = bias ? (double)bias[c] : 0.0;
            for (int kh = 0; kh < g->KH; kh++)
                for (int kw = 0; kw < g->KW; kw++)
                    s += (double)W[((int64_t)c * g->KH + kh) * g->KW + kw] *
                         x_at(x, g, b, oh * g->sh - g->ph + kh * g->dh, ow * g->sw - g->pw + kw * g->dw, c);
            y[p * g->C_in + c] = act(s, g->relu);
        }
    }
}

/* ------------------------------------------------------------------ */
/* Fine-tuning with the mask held fixed (Sec. 3.2 keeps the selected    */
/* blocks and Sec. 4.1 fine-tunes the pruned network; the pruned blocks  */
/* stay zero): the gradients of Eq. 6's pre-activation output y with     */
/* respect to the input and to the kept weights, from dy = dL/dy          */
/* [B][Ho][Wo][C_out].  Written from the definition of y:                */
/*   dx[b,ih,iw,c] = sum over (o, kh, kw, oh, ow) with                    */
/*                   oh*sh - ph + kh*dh = ih and ow*sw - pw + kw*dw = iw   */
/*                   of mask * W[o,c,kh,kw] * dy[b,oh,ow,o]               */
/*   dW[o,c,kh,kw] = mask * sum_{b,oh,ow} dy[b,oh,ow,o]                   */
/*                   * x[b, oh*sh - ph + kh*dh, ow*sw - pw + kw*dw, c]     */
/* (zero padding: positions outside the image contribute nothing).       */
/* absacc (nullable) = the same sums over |terms|.                       */
/* ------------------------------------------------------------------ */
static double dy_at(const float *dy, const oracle_geom *g, int Ho, int Wo, int b, int oh, int ow, int o)
{
    return (double)dy[(((int64_t)b * Ho + oh) * Wo + ow) * g->C_out + o];
}

void oracle_conv_backward_data(const float *dy, const float *W, const uint8_t *mask,
                               const oracle_geom *g, int N, double *dx, double *absacc)
{
    int Ho = out_size(g->H, g->KH, g->sh, g->ph, g->dh);
    int Wo = out_size(g->W, g->KW, g->sw, g->pw, g->dw);
    int K = g->KH * g->KW * g->C_in;
    int64_t total = (int64_t)g->B * g->H * g->W;
#pragma omp parallel for schedule(dynamic, 16)
    for (int64_t q = 0; q < total; q++) {
        int b = (int)(q / ((int64_t)g->H * g->W));
        int ih = (int)((q / g->W) % g->H), iw = (int)(q % g->W);
        for (int c = 0; c < g->C_in; c++) {
            double s = 0.0, a = 0.0;
            for (int kh = 0; kh < g->KH; kh++) {
                int th = ih + g->ph - kh * g->dh;          /* = oh * sh */
                if (th < 0 || th % g->sh != 0 || th / g->sh >= Ho) continue;
                for (int kw = 0; kw < g->KW; kw++) {
                    int tw = iw + g->pw - kw * g->dw;      /* = ow * sw */
                    if (tw < 0 || tw % g->sw != 0 || tw / g->sw >= Wo) continue;
                    int k = (kh * g->KW + kw) * g->C_in + c;
                    for (int o = 0; o < g->C_out; o++) {
                        if (mask && !mask[(int64_t)(o / N) * K + k]) continue;
                        double t = w_at(W, g->C_in, g->KH, g->KW, o, c, kh, kw) *
                                   dy_at(dy, g, Ho, Wo, b, th / g->sh, tw / g->sw, o);
                        s += t;
                        a += fabs(t);
                    }
                }
            }
            dx[q * g->C_in + c] = s;
            if (absacc) absacc[q * g->C_in + c] = a;
        }
    }
}

void oracle_conv_backward_weight(const float *x, const float *dy, const uint8_t *mask,
                                 const oracle_geom *g, int N, double *dW, double *absacc)
{
    int Ho = out_size(g->H, g->KH, g->sh, g->ph, g->dh);
    int Wo = out_size(g->W, g->KW, g->sw, g->pw, g->dw);
    int K = g->KH * g->KW * g->C_in;
#pragma omp parallel for schedule(dynamic, 1)
    for (int o = 0; o < g->C_out; o++)
        for (int c = 0; c < g->C_in; c++)
            for (int kh = 0; kh < g->KH; kh++)
                for (int kw = 0; kw < g->KW; kw++) {
                    int k = (kh * g->KW + kw) * g->C_in + c;
                    int64_t at = (((int64_t)o * g->C_in + c) * g->KH + kh) * g->KW + kw;
                    double s = 0.0, a = 0.0;
                    if (!mask || mask[(int64_t)(o / N) * K + k])
                        for (int b = 0; b < g->B; b++)
                            for (int oh = 0; oh < Ho; oh++)
                                for (int ow = 0; ow < Wo; ow++) {
                                    double t = dy_at(dy, g, Ho, Wo, b, oh, ow, o) *
                                               x_at(x, g, b, oh * g->sh - g->ph + kh * g->dh,
                                                    ow * g->sw - g->pw + kw * g->dw, c);
                                    s += t;
                                    a += fabs(t);
                                }
                    dW[at] = s;
                    if (absacc) absacc[at] = a;
                }
}

int oracle_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
